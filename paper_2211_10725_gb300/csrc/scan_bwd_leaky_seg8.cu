// 8-step segments of the register-segment recompute BPTT (scan_seg.cuh),
// every instantiated dtype pair.
#include "scan_seg_launch.cuh"

namespace snn {

cudaError_t launch_scan_bwd_leaky_seg_k8(ScanArgs a, int in_dt, int io_dt, cudaStream_t stream,
                                         bool* launched) {
  SNN_DTYPE_DISPATCH(in_dt, io_dt, return (seg_launch::seg_modes<TI, TO, 8>(a, stream, launched)));
}

}  // namespace snn
