// 12-step segments of the register-segment recompute BPTT (scan_seg.cuh)
// for half-precision inputs: 12 rows of 4 lanes = 48 trace registers a
// thread, checkpoint traffic 2/3 of the 8-step segments'.
#include "scan_seg_launch.cuh"

namespace snn {

cudaError_t launch_scan_bwd_leaky_seg_k12(ScanArgs a, int in_dt, int io_dt, cudaStream_t stream,
                                          bool* launched) {
  if (in_dt == 1 && io_dt == 1) {
    return seg_launch::seg_modes<__nv_bfloat16, __nv_bfloat16, 12>(a, stream, launched);
  }
  if (in_dt == 2 && io_dt == 2) return seg_launch::seg_modes<__half, __half, 12>(a, stream, launched);
  return cudaSuccess;
}

}  // namespace snn
