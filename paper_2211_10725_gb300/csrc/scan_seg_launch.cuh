// Launch templates of the register-segment recompute BPTT (scan_seg.cuh),
// shared by the translation units that instantiate its checkpoint
// intervals.
#pragma once

#include "scan_dispatch.cuh"
#include "scan_seg.cuh"

namespace snn {
namespace seg_launch {

template <typename TI, typename TO, int RESET, int SG, int KC, bool REC>
cudaError_t seg(ScanArgs a, cudaStream_t st, bool* launched) {
  const void* k = (const void*)scan_bwd_seg<TI, TO, RESET, SG, KC, REC>;
  constexpr int RH = KC < kSegItemRows ? KC : kSegItemRows;
  const int replay = 4 + RH * (int)sizeof(TI);                // checkpoint + RH rows of I
  const int grad = RH * (int)sizeof(TO);                      // RH rows of grad_spk
  StagedPlan p;
  if (!plan_staged(k, a.L, 2 * (int64_t)a.nseg * (KC / RH), replay > grad ? replay : grad, 0,
                   kSegLanes<KC>, &p))
    return cudaSuccess;
  a.lanes_per_cta = p.lanes_per_cta;
  a.stages = p.stages;
  a.stage_bytes = p.stage_bytes;
  *launched = true;
  return launch_pdl(scan_bwd_seg<TI, TO, RESET, SG, KC, REC>, dim3((unsigned)p.grid),
                    dim3(p.threads), p.smem, st, a);
}

template <typename TI, typename TO, int KC>
cudaError_t seg_modes(ScanArgs a, cudaStream_t st, bool* launched) {
  const bool atan = a.sg == SG_ATAN;
  if (a.rec)
    return atan ? seg<TI, TO, RESET_SUBTRACT, SG_ATAN, KC, true>(a, st, launched)
                : seg<TI, TO, RESET_SUBTRACT, SG_FAST_SIGMOID, KC, true>(a, st, launched);
  if (a.reset == RESET_SUBTRACT)
    return atan ? seg<TI, TO, RESET_SUBTRACT, SG_ATAN, KC, false>(a, st, launched)
                : seg<TI, TO, RESET_SUBTRACT, SG_FAST_SIGMOID, KC, false>(a, st, launched);
  if (a.reset == RESET_ZERO)
    return atan ? seg<TI, TO, RESET_ZERO, SG_ATAN, KC, false>(a, st, launched)
                : seg<TI, TO, RESET_ZERO, SG_FAST_SIGMOID, KC, false>(a, st, launched);
  return cudaSuccess;  // no reset: the general kernel
}

}  // namespace seg_launch

// One checkpoint interval's dtype dispatch (scan_bwd_leaky_seg*.cu).
cudaError_t launch_scan_bwd_leaky_seg_k8(ScanArgs a, int in_dt, int io_dt, cudaStream_t stream,
                                         bool* launched);
cudaError_t launch_scan_bwd_leaky_seg_k12(ScanArgs a, int in_dt, int io_dt, cudaStream_t stream,
                                          bool* launched);
cudaError_t launch_scan_bwd_leaky_seg_k16(ScanArgs a, int in_dt, int io_dt, cudaStream_t stream,
                                          bool* launched);

}  // namespace snn
