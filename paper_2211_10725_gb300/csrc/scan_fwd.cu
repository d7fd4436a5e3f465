// Forward scan launchers (Leaky and Synaptic).
#include "scan_dispatch.cuh"

namespace snn {

cudaError_t launch_scan_fwd(ScanArgs a, bool synaptic, int in_dt, int io_dt, bool staged,
                            cudaStream_t stream) {
  if (synaptic) SNN_DTYPE_DISPATCH(in_dt, io_dt, return (fwd_t<true, TI, TO>(a, staged, stream)));
  SNN_DTYPE_DISPATCH(in_dt, io_dt, return (fwd_t<false, TI, TO>(a, staged, stream)));
}

}  // namespace snn
