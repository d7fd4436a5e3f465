// BPTT launchers for the Leaky neuron, recompute variant (checkpointed
// replay of the forward inside the reverse pass).
#include "scan_dispatch.cuh"

namespace snn {

cudaError_t launch_scan_bwd_leaky_recompute(ScanArgs a, int in_dt, int io_dt, bool staged,
                                            cudaStream_t stream) {
  bool launched = false;
  const cudaError_t e = launch_scan_bwd_leaky_seg(a, in_dt, io_dt, staged, stream, &launched);
  if (launched || e != cudaSuccess) return e;
  SNN_DTYPE_DISPATCH(in_dt, io_dt, return (bwd_t<false, true, TI, TO>(a, staged, stream)));
}

}  // namespace snn
