// Launchers of the register-segment recompute BPTT (scan_seg.cuh) for the
// Leaky and recurrent Leaky neurons: 16-step segments here, 8- and 12-step
// ones in scan_bwd_leaky_seg8.cu and scan_bwd_leaky_seg12.cu (separate
// translation units compile in parallel).
#include "scan_seg_launch.cuh"

namespace snn {

cudaError_t launch_scan_bwd_leaky_seg_k16(ScanArgs a, int in_dt, int io_dt, cudaStream_t stream,
                                          bool* launched) {
  // 16-step segments for half-precision inputs only (16 rows of 4 lanes =
  // 32 registers per thread; fp32 rows would double that)
  if (in_dt == 1 && io_dt == 1) {
    return seg_launch::seg_modes<__nv_bfloat16, __nv_bfloat16, 16>(a, stream, launched);
  }
  if (in_dt == 2 && io_dt == 2) return seg_launch::seg_modes<__half, __half, 16>(a, stream, launched);
  return cudaSuccess;
}

cudaError_t launch_scan_bwd_leaky_seg(ScanArgs a, int in_dt, int io_dt, bool staged,
                                      cudaStream_t stream, bool* launched) {
  *launched = false;
  if (!staged || a.L == 0 || a.T == 0 || (a.debug & DEBUG_NO_SEGMENT)) return cudaSuccess;
  if (a.gm || a.L % 8 != 0) return cudaSuccess;  // per-step dL/dmem: the general kernel
  if (a.K == 8) return launch_scan_bwd_leaky_seg_k8(a, in_dt, io_dt, stream, launched);
  if (a.K == 12) return launch_scan_bwd_leaky_seg_k12(a, in_dt, io_dt, stream, launched);
  if (a.K == 16) return launch_scan_bwd_leaky_seg_k16(a, in_dt, io_dt, stream, launched);
  return cudaSuccess;
}

}  // namespace snn
