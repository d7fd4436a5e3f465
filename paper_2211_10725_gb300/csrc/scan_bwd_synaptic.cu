// BPTT launchers for the Synaptic neuron: the store variant here, the
// recompute variant in scan_bwd_synaptic_recompute.cu (separate translation
// units compile in parallel).
#include "scan_dispatch.cuh"

namespace snn {

cudaError_t launch_scan_bwd_synaptic(ScanArgs a, bool recompute, int in_dt, int io_dt,
                                     bool staged, cudaStream_t stream) {
  if (recompute) return launch_scan_bwd_synaptic_recompute(a, in_dt, io_dt, staged, stream);
  SNN_DTYPE_DISPATCH(in_dt, io_dt, return (bwd_t<true, false, TI, TO>(a, staged, stream)));
}

}  // namespace snn
