// BPTT launchers for the Synaptic neuron, recompute variant (checkpointed
// replay of the forward inside the reverse pass).
#include "scan_dispatch.cuh"

namespace snn {

cudaError_t launch_scan_bwd_synaptic_recompute(ScanArgs a, int in_dt, int io_dt, bool staged,
                                               cudaStream_t stream) {
  SNN_DTYPE_DISPATCH(in_dt, io_dt, return (bwd_t<true, true, TI, TO>(a, staged, stream)));
}

}  // namespace snn
