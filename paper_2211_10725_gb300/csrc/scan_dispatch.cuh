// Templated launchers for the scan kernels; each .cu file instantiates one
// family so the library compiles in parallel.
#pragma once

#include <type_traits>

#include "scan_host.cuh"

namespace snn {

// dtype pairs (input, io) whose staged backward gets loops specialised on
// the reset mode and surrogate; other pairs use the run-time-mode loop.
template <typename TI, typename TO>
constexpr bool kSpecialise =
    (std::is_same<TI, float>::value && std::is_same<TO, float>::value) ||
    (std::is_same<TI, __nv_bfloat16>::value && std::is_same<TO, __nv_bfloat16>::value) ||
    (std::is_same<TI, float>::value && std::is_same<TO, __nv_bfloat16>::value);

template <bool SYN, typename TI, typename TO, int RESET, bool REC = false>
cudaError_t fwd_staged(ScanArgs a, cudaStream_t st, bool* launched) {
  const void* k = (const void*)scan_fwd_staged<SYN, TI, TO, RESET, REC>;
  StagedPlan p;
  // a stage holds kFwdRows steps of the strip's input row; one CTA per SM
  // where it fits (the longer rows stream faster), two for short sequences
  // (T <= 64: a CTA's few stages fill and drain while the SM's other CTA
  // computes; measured 2-4% faster at T = 25, 0.5% slower at T = 500)
  if (!plan_staged(k, a.L, ceil_div(a.T, kFwdRows), kFwdRows * (int)sizeof(TI), 0, kLanes<SYN>, &p,
                   0, 0, a.T <= 64 ? 2 : 1))
    return cudaSuccess;
  a.lanes_per_cta = p.lanes_per_cta;
  a.stages = p.stages;
  a.stage_bytes = p.stage_bytes;
  *launched = true;
  return launch_pdl(scan_fwd_staged<SYN, TI, TO, RESET, REC>, dim3((unsigned)p.grid),
                    dim3(p.threads), p.smem, st, a);
}

template <bool SYN, typename TI, typename TO>
cudaError_t fwd_t(ScanArgs a, bool staged, cudaStream_t st) {
  if (staged && a.L > 0) {
    bool launched = false;
    cudaError_t e;
    if (!SYN && a.rec) e = fwd_staged<false, TI, TO, RESET_SUBTRACT, true>(a, st, &launched);
    else if (a.reset == RESET_SUBTRACT) e = fwd_staged<SYN, TI, TO, RESET_SUBTRACT>(a, st, &launched);
    else if (a.reset == RESET_ZERO) e = fwd_staged<SYN, TI, TO, RESET_ZERO>(a, st, &launched);
    else e = fwd_staged<SYN, TI, TO, -1>(a, st, &launched);
    if (launched || e != cudaSuccess) return e;
  }
  if (a.L == 0) return cudaSuccess;
  return launch_pdl(scan_fwd_plain<SYN, TI, TO>, dim3((unsigned)ceil_div(a.L, 256)), dim3(256), 0,
                    st, a);
}

template <bool SYN, bool RECOMP, typename TI, typename TO, int RESET, int SG, int KC, bool REC,
          int VL>
cudaError_t bwd_staged_vl(ScanArgs a, cudaStream_t st, bool* launched) {
  const void* k = (const void*)scan_bwd_staged<SYN, RECOMP, TI, TO, RESET, SG, KC, REC, VL>;
  int per_lane, seg, fixed;
  int64_t items;
  if (RECOMP) {
    const int fwd_item = (int)sizeof(TI);
    const int bwd_item = (int)sizeof(TO) * (a.gm ? 2 : 1);
    per_lane = fwd_item > bwd_item ? fwd_item : bwd_item;
    seg = kLanes<SYN> * 4 * a.K * (SYN ? 2 : 1);
    fixed = 2 * 4 * (SYN ? 2 : 1);  // two checkpoint slots
    items = 2 * a.T;
  } else {
    const int n = 2 + (sizeof(TO) != 4 ? 1 : 0) + ((SYN && a.part_alpha) ? 1 : 0) + (a.gm ? 1 : 0);
    per_lane = n * (int)sizeof(TO);
    seg = 0;
    fixed = 0;
    items = a.T;
  }
  StagedPlan p;
  if (!plan_staged(k, a.L, items, per_lane, seg, VL, &p, fixed, KC)) return cudaSuccess;
  a.lanes_per_cta = p.lanes_per_cta;
  a.stages = p.stages;
  a.stage_bytes = p.stage_bytes;
  *launched = true;
  return launch_pdl(scan_bwd_staged<SYN, RECOMP, TI, TO, RESET, SG, KC, REC, VL>,
                    dim3((unsigned)p.grid), dim3(p.threads), p.smem, st, a);
}

// The staged backward with its lanes per thread: 4 for the Leaky neuron's
// store mode on sequences of at most 64 steps, else kLanes.
template <bool SYN, bool RECOMP, typename TI, typename TO, int RESET, int SG, int KC = 0,
          bool REC = false>
cudaError_t bwd_staged(ScanArgs a, cudaStream_t st, bool* launched) {
  if constexpr (!SYN && !RECOMP) {
    if (a.T <= 64) return bwd_staged_vl<SYN, RECOMP, TI, TO, RESET, SG, KC, REC, 4>(a, st, launched);
  }
  return bwd_staged_vl<SYN, RECOMP, TI, TO, RESET, SG, KC, REC, kLanes<SYN>>(a, st, launched);
}

template <bool SYN, bool RECOMP, typename TI, typename TO>
cudaError_t bwd_t(ScanArgs a, bool staged, cudaStream_t st) {
  if (staged && a.L > 0) {
    bool launched = false;
    cudaError_t e = cudaSuccess;
    bool done = false;
    if (!SYN && a.rec) {  // recurrent Leaky neuron: reset by subtraction (Eq. 7)
      if constexpr (kSpecialise<TI, TO>) {
        if (a.sg == SG_ATAN)
          e = bwd_staged<false, RECOMP, TI, TO, RESET_SUBTRACT, SG_ATAN, 0, true>(a, st, &launched);
        else
          e = bwd_staged<false, RECOMP, TI, TO, RESET_SUBTRACT, SG_FAST_SIGMOID, 0, true>(a, st,
                                                                                      &launched);
      } else {
        e = bwd_staged<false, RECOMP, TI, TO, RESET_SUBTRACT, -1, 0, true>(a, st, &launched);
      }
      done = true;
    } else if constexpr (kSpecialise<TI, TO>) {
      done = true;
      const int key = (a.reset == RESET_NONE ? 9 : a.reset * 2 + a.sg);
      // the recompute variant with the default checkpoint interval K = 8
      // also has a fully unrolled segment body (ring of exactly 8 stages)
      const bool k8 = RECOMP && a.K == 8;
      switch (key) {
        case 0:
          if (k8) e = bwd_staged<SYN, RECOMP, TI, TO, RESET_SUBTRACT, SG_FAST_SIGMOID, 8>(a, st, &launched);
          if (!launched && e == cudaSuccess)
            e = bwd_staged<SYN, RECOMP, TI, TO, RESET_SUBTRACT, SG_FAST_SIGMOID>(a, st, &launched);
          break;
        case 1:
          if (k8) e = bwd_staged<SYN, RECOMP, TI, TO, RESET_SUBTRACT, SG_ATAN, 8>(a, st, &launched);
          if (!launched && e == cudaSuccess)
            e = bwd_staged<SYN, RECOMP, TI, TO, RESET_SUBTRACT, SG_ATAN>(a, st, &launched);
          break;
        case 2: e = bwd_staged<SYN, RECOMP, TI, TO, RESET_ZERO, SG_FAST_SIGMOID>(a, st, &launched); break;
        case 3: e = bwd_staged<SYN, RECOMP, TI, TO, RESET_ZERO, SG_ATAN>(a, st, &launched); break;
        default: done = false;
      }
    }
    if (!done) e = bwd_staged<SYN, RECOMP, TI, TO, -1, -1>(a, st, &launched);
    if (launched || e != cudaSuccess) return e;
  }
  if (a.L == 0) return cudaSuccess;
  const int threads = 128;
  const size_t smem = RECOMP ? (size_t)a.K * threads * 4 * (SYN ? 2 : 1) : 0;
  const void* k = (const void*)scan_bwd_plain<SYN, RECOMP, TI, TO>;
  cudaError_t e = ensure_smem(k, smem);
  if (e != cudaSuccess) return e;
  return launch_pdl(scan_bwd_plain<SYN, RECOMP, TI, TO>, dim3((unsigned)ceil_div(a.L, threads)),
                    dim3(threads), smem, st, a);
}

// dtype codes (snn_dtype_t): 0 f32, 1 bf16, 2 f16.  Instantiated pairs
// (in, io): (f32,f32) (bf16,bf16) (f16,f16) (f32,bf16) (f32,f16).
#define SNN_DTYPE_DISPATCH(IN_DT, IO_DT, CALL)                                   \
  do {                                                                           \
    if ((IN_DT) == 0 && (IO_DT) == 0) { using TI = float; using TO = float; CALL; } \
    if ((IN_DT) == 1 && (IO_DT) == 1) { using TI = __nv_bfloat16; using TO = __nv_bfloat16; CALL; } \
    if ((IN_DT) == 2 && (IO_DT) == 2) { using TI = __half; using TO = __half; CALL; } \
    if ((IN_DT) == 0 && (IO_DT) == 1) { using TI = float; using TO = __nv_bfloat16; CALL; } \
    if ((IN_DT) == 0 && (IO_DT) == 2) { using TI = float; using TO = __half; CALL; } \
    return cudaErrorNotSupported;                                                \
  } while (0)

}  // namespace snn
