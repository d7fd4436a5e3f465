// BPTT launchers for the Synaptic neuron (store and recompute variants).
#include "scan_dispatch.cuh"

namespace snn {

cudaError_t launch_scan_bwd_synaptic(ScanArgs a, bool recompute, int in_dt, int io_dt,
                                     bool staged, cudaStream_t stream) {
  if (recompute) SNN_DTYPE_DISPATCH(in_dt, io_dt, return (bwd_t<true, true, TI, TO>(a, staged, stream)));
  SNN_DTYPE_DISPATCH(in_dt, io_dt, return (bwd_t<true, false, TI, TO>(a, staged, stream)));
}

}  // namespace snn
