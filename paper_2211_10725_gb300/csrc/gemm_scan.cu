// Dense layer with the Leaky scan in its epilogue: the synaptic operation
// w.x of Fig. 3 for every time step as one tcgen05 GEMM, and Eq. (4) run on
// the accumulator before it ever reaches HBM.
//
// The rows of the layer input are (t, r): X [T, R, K] with R = B*P (P > 1:
// the pixels of a convolution's patch rows).  A work tile is BS rows r for
// all T steps (BS*T <= 128): one 3-D TMA box {64 of K, BS rows, T steps}
// lands as BS*T 128-byte rows ordered (t, r), which is the MMA's A tile, so
// a tile's accumulator holds whole time series of BS*BN lanes.
//
// Warp roles as in the plain GEMM (warp 0 TMA, warp 1 MMA into two TMEM
// accumulators).  Warps 2-5 copy a finished accumulator to shared memory
// (fp32, rows padded against bank conflicts) and hand it back to the MMA
// warp; then warps 2-11 scan: each thread owns lanes (r, n) and steps them
// through t with the same fwd_step the scan kernels use (one rounded fp32
// operation at a time, bit-identical to them), writing spk and the bf16
// membrane trace [T, R, N] and, optionally, the spike bits the store-mode
// BPTT reads (bit k of byte j of row t is z_t of lane 8j + k).  The fp32
// current is never written.
//
// Backward mode (BWD): the same tiles of the product dX = dI_up * W (W read
// MN-major, as the plain dense backward reads it) are the spike gradients
// dL/dz of the layer below, and the epilogue runs that layer's BPTT on them
// in reverse time with the scan kernels' bwd_step, from its stored bf16
// trace and spike bits, writing its dL/dI.  The spike gradient is never
// rounded or written.
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include <climits>
#include <cstdint>

#include "snn.h"
#include "tcgen05.cuh"

namespace snn {
namespace gemm {
namespace {

constexpr int kFusedStages = 3;  // with BN <= 64, two CTAs fit on an SM
constexpr int kScanWarps = 10;  // warps 2..11 scan; 2..5 also drain the accumulator
constexpr int kScanThreads = 32 * kScanWarps;
constexpr int kFusedThreads = 64 + kScanThreads;
constexpr int kScanLanes = 2;  // lanes a scan thread steps together (independent chains)
constexpr int kBwdChunk = 8;   // steps of stored trace a backward scan thread loads ahead

struct FusedArgs {
  int T, R, K, N;   // steps, rows per step, reduction, output columns (neurons / channels)
  int BS;           // rows r per tile
  int reset;
  int beta_col, thr_col;  // 1: one value per output column, 0: scalar
  const float* beta;
  const float* thr;
  __nv_bfloat16* spk;  // [T, R, N]
  __nv_bfloat16* mem;
  unsigned char* bits;  // or null
  int64_t bits_row;
  int* status;
  uint64_t wait_ns;
  // backward mode: the layer's stored trace, spike bits (or spk) and dL/dI
  const __nv_bfloat16* mem_in;
  const unsigned char* bits_in;
  const __nv_bfloat16* spk_in;
  __nv_bfloat16* gI;
  ScanArgs sa;  // reset, detach and surrogate of bwd_step
};

template <int BN>
__host__ __device__ constexpr int stage_pitch() { return BN + 4; }  // floats per staged row

template <int BN>
__host__ __device__ constexpr size_t fused_smem_bytes() {
  return 1024 + (size_t)kFusedStages * (BM * BK * 2 + BN * BK * 2) +
         (size_t)BM * stage_pitch<BN>() * 4 + 256;  // barriers, TMEM slot, wait flags
}

__device__ __forceinline__ void epi_barrier() {
  asm volatile("bar.sync 1, %0;" ::"n"(kScanThreads) : "memory");
}

template <int BN, int RESET, bool BWD = false, int SG = 0>
__global__ void __launch_bounds__(kFusedThreads, 2)
    gemm_leaky_tcgen05(const __grid_constant__ CUtensorMap ta, const __grid_constant__ CUtensorMap tb,
                       const FusedArgs f) {
  static_assert(BN % 16 == 0 && BN >= 16 && BN <= 128, "UMMA N for M=128");
  static_assert(!BWD || BN % 64 == 0, "an MN-major B tile is whole 64-wide boxes");
  constexpr int A_BYTES = BM * BK * 2;
  constexpr int B_BYTES = BN * BK * 2;
  constexpr int SP = stage_pitch<BN>();
  constexpr uint32_t TCOLS = tmem_cols<BN>();
  constexpr int kEpiWarps = 4;
  extern __shared__ unsigned char smem_raw[];
  unsigned char* smem =
      reinterpret_cast<unsigned char*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  unsigned char* sA = smem;
  unsigned char* sB = smem + kFusedStages * A_BYTES;
  float* stg = reinterpret_cast<float*>(sB + kFusedStages * B_BYTES);  // [128][SP]
  uint64_t* full = reinterpret_cast<uint64_t*>(stg + BM * SP);
  uint64_t* empty = full + kFusedStages;
  uint64_t* acc_full = empty + kFusedStages;
  uint64_t* acc_empty = acc_full + 2;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(acc_empty + 2);
  int* epi_ok = reinterpret_cast<int*>(tmem_slot + 1);  // [4] per epilogue warp: its wait succeeded
  const int warp = threadIdx.x >> 5, lid = threadIdx.x & 31;
  const int nk = (f.K + BK - 1) / BK;
  const int tiles_n = (f.N + BN - 1) / BN;
  const int tiles = tiles_n * ((f.R + f.BS - 1) / f.BS);
  const uint32_t a_tx = (uint32_t)(f.BS * f.T * 128);  // bytes of one A box

  if (threadIdx.x == 0) {
    for (int s = 0; s < kFusedStages; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(&acc_full[b], 1);
      mbar_init(&acc_empty[b], kEpiWarps);
    }
    fence_barrier_init();
  }
  if (warp == 1) tmem_alloc(tmem_slot, TCOLS);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  grid_dep_wait();

  if (warp == 0) {
    if (lid == 0) {
      int64_t n_issued = 0;
      bool ok = true;
      for (int t = blockIdx.x; t < tiles && ok; t += gridDim.x) {
        const int r0 = (t / tiles_n) * f.BS, n0 = (t % tiles_n) * BN;
        for (int kb = 0; kb < nk; ++kb, ++n_issued) {
          const int s = (int)(n_issued % kFusedStages);
          if (n_issued >= kFusedStages &&
              !mbar_wait_poll(&empty[s], (uint32_t)(((n_issued / kFusedStages) - 1) & 1), f.wait_ns)) {
            record_status(f.status, kStatusTimeout);
            ok = false;
            break;
          }
          mbar_arrive_expect_tx(&full[s], a_tx + B_BYTES);
          tma_load_3d(sA + s * A_BYTES, &ta, kb * BK, r0, 0, &full[s]);
          if constexpr (BWD) {
#pragma unroll
            for (int j = 0; j < BN / 64; ++j)
              tma_load_2d(sB + s * B_BYTES + j * kMnBoxBytes, &tb, n0 + 64 * j, kb * BK, &full[s]);
          } else {
            tma_load_2d(sB + s * B_BYTES, &tb, kb * BK, n0, &full[s]);
          }
        }
      }
      for (int64_t j = n_issued > kFusedStages ? n_issued - kFusedStages : 0; j < n_issued; ++j)
        mbar_wait_bounded(&full[j % kFusedStages], (uint32_t)((j / kFusedStages) & 1), kDrainWaitNs);
    }
  } else if (warp == 1) {
    if (lid == 0) {
      constexpr uint32_t idesc = idesc_bf16(BM, BN, false, BWD);
      // 16 more along K: 32 bytes inside a K-major row, or 16 rows (2048
      // bytes) of an MN-major tile; the descriptor holds the address >> 4
      constexpr uint64_t stepB = BWD ? 2048 >> 4 : 32 >> 4;
      int64_t n_used = 0;
      bool ok = true;
      int i = 0;
      for (int t = blockIdx.x; t < tiles && ok; t += gridDim.x, ++i) {
        const int b = i & 1;
        if (i >= 2 && !mbar_wait_poll(&acc_empty[b], (uint32_t)(((i >> 1) - 1) & 1), f.wait_ns)) {
          record_status(f.status, kStatusTimeout);
          break;
        }
        tc_fence_after();
        const uint32_t acc = tmem + (uint32_t)(b * BN);
        for (int kb = 0; kb < nk; ++kb, ++n_used) {
          const int s = (int)(n_used % kFusedStages);
          if (!mbar_wait_poll(&full[s], (uint32_t)((n_used / kFusedStages) & 1), f.wait_ns)) {
            record_status(f.status, kStatusTimeout);
            ok = false;
            break;
          }
          tc_fence_after();
          const uint64_t da = sdesc_sw128(sA + s * A_BYTES);
          const uint64_t db = BWD ? sdesc_sw128_mn(sB + s * B_BYTES) : sdesc_sw128(sB + s * B_BYTES);
#pragma unroll
          for (int kk = 0; kk < BK / 16; ++kk)
            tc_mma(acc, da + (uint64_t)(2 * kk), db + stepB * kk, idesc, (kb | kk) != 0 ? 1u : 0u);
          tc_commit(&empty[s]);
        }
        if (ok) tc_commit(&acc_full[b]);
      }
    }
  } else {
    const int q = warp & 3;          // TMEM lane quarter of a draining warp (warps 2..5)
    const bool drains = warp < 6;
    const int e = threadIdx.x - 64;  // 0..kScanThreads-1 among the scan threads
    const int lanes = f.BS * BN;
    int i = 0;
    for (int t = blockIdx.x; t < tiles; t += gridDim.x, ++i) {
      const int b = i & 1;
      const bool waited =
          drains ? warp_wait_uniform(&acc_full[b], (uint32_t)((i >> 1) & 1), f.wait_ns) : true;
      const int r0 = (t / tiles_n) * f.BS, n0 = (t % tiles_n) * BN;
      if (drains && waited) {
        tc_fence_after();
        // accumulator -> shared memory: row = TMEM lane = (t, r) of the tile
        const uint32_t acc = tmem + ((uint32_t)(q * 32) << 16) + (uint32_t)(b * BN);
        float* srow = stg + (q * 32 + lid) * SP;
#pragma unroll 1
        for (int c = 0; c < BN; c += 16) {
          uint32_t r[16];
          tmem_ld16(acc + (uint32_t)c, r);
#pragma unroll
          for (int j = 0; j < 4; ++j)
            *reinterpret_cast<float4*>(srow + c + 4 * j) =
                make_float4(__uint_as_float(r[4 * j]), __uint_as_float(r[4 * j + 1]),
                            __uint_as_float(r[4 * j + 2]), __uint_as_float(r[4 * j + 3]));
        }
        tc_fence_before();
        __syncwarp();
        if (lid == 0) mbar_arrive(&acc_empty[b]);  // the MMA may refill this accumulator
      }
      if (drains && lid == 0) epi_ok[q] = waited ? 1 : 0;
      epi_barrier();  // every row is staged, and every warp's wait result is known
      if (!(epi_ok[0] && epi_ok[1] && epi_ok[2] && epi_ok[3])) {  // the same answer in all four warps
        if (e == 0) record_status(f.status, kStatusTimeout);
        break;
      }
      if constexpr (BWD) {
        // the reverse scan: thread e steps lanes j = g0 + e from t = T-1 down
        // to 0; the staged value of (t, lane) is dL/dz_t.  The stored trace
        // comes in chunks of kBwdChunk steps, the next chunk's loads issued
        // before the current chunk is stepped, so a lane waits for memory
        // about once rather than once per step.
        const int64_t RN = (int64_t)f.R * f.N;
        for (int g0 = 0; g0 < lanes; g0 += kScanThreads) {
          const int j = g0 + e;
          const int jj = j < lanes ? j : 0;  // lanes past the tile read row 0
          const int sr = jj / BN, n = jj - (jj / BN) * BN;
          const bool ok = j < lanes && r0 + sr < f.R && n0 + n < f.N;
          const int nc = ok ? n0 + n : 0;
          const float beta = __ldg(f.beta + (f.beta_col ? nc : 0));
          const float thr = __ldg(f.thr + (f.thr_col ? nc : 0));
          const int64_t o = ok ? (int64_t)(r0 + sr) * f.N + nc : 0;
          const float* gsp = stg + sr * SP + n;
          BwdLane st{0.0f, 0.0f, 0.0f, 0.0f, 0.0f};
          // chunk at tc: steps tc, tc-1, ..., tc-kBwdChunk+1; steps before 0
          // load step 0 (in bounds) and are not stepped
          auto load_chunk = [&](int tc, __nv_bfloat16 (&u)[kBwdChunk], uint32_t& zm) {
            zm = 0;
#pragma unroll
            for (int c = 0; c < kBwdChunk; ++c) {
              const int ts = tc - c >= 0 ? tc - c : 0;
              const int64_t q = (int64_t)ts * RN + o;
              u[c] = f.mem_in[q];
              const uint32_t z =
                  f.bits_in ? (__ldg(f.bits_in + (int64_t)ts * f.bits_row + (o >> 3)) >> (o & 7)) & 1u
                            : (__bfloat162float(f.spk_in[q]) != 0.0f ? 1u : 0u);
              zm |= z << c;
            }
          };
          __nv_bfloat16 ucur[kBwdChunk], unext[kBwdChunk];
          uint32_t zcur, znext = 0;
          load_chunk(f.T - 1, ucur, zcur);
          for (int tc = f.T - 1; tc >= 0; tc -= kBwdChunk) {
            if (tc - kBwdChunk >= 0) load_chunk(tc - kBwdChunk, unext, znext);
#pragma unroll
            for (int c = 0; c < kBwdChunk; ++c) {
              const int ts = tc - c;
              if (ts < 0) break;
              const float du =
                  bwd_step<false, RESET, SG>(f.sa, beta, thr, 0.0f, ts + 1 < f.T, __bfloat162float(ucur[c]),
                                             ((zcur >> c) & 1u) != 0, 0.0f, gsp[ts * f.BS * SP], 0.0f, 0.0f, st);
              if (ok) f.gI[(int64_t)ts * RN + o] = __float2bfloat16_rn(du);
            }
#pragma unroll
            for (int c = 0; c < kBwdChunk; ++c) ucur[c] = unext[c];
            zcur = znext;
          }
        }
      } else {
        // the scan: thread e steps lanes j = g0 + kScanThreads*v + e together
        // (independent chains); groups wholly past the tile are skipped
        const int64_t RN = (int64_t)f.R * f.N;  // elements per step of spk / mem
        for (int g0 = 0; g0 < lanes; g0 += kScanThreads * kScanLanes) {
          const int nv = (lanes - g0 + kScanThreads - 1) / kScanThreads;  // block-uniform
          float u[kScanLanes], beta[kScanLanes], thr[kScanLanes];
          bool z[kScanLanes], ok[kScanLanes];
          const float* xs[kScanLanes];
          __nv_bfloat16* ps[kScanLanes];
          __nv_bfloat16* pm[kScanLanes];
          unsigned char* pb[kScanLanes];
#pragma unroll
          for (int v = 0; v < kScanLanes; ++v) {
            const int j = g0 + kScanThreads * v + e;
            const int jj = j < lanes ? j : 0;  // lanes past the tile read row 0
            const int s = jj / BN, n = jj - (jj / BN) * BN;
            ok[v] = j < lanes && r0 + s < f.R && n0 + n < f.N;
            const int nc = ok[v] ? n0 + n : 0;
            beta[v] = __ldg(f.beta + (f.beta_col ? nc : 0));
            thr[v] = __ldg(f.thr + (f.thr_col ? nc : 0));
            u[v] = 0.0f;
            z[v] = false;
            const int64_t o = ok[v] ? (int64_t)(r0 + s) * f.N + nc : 0;  // lane index within a step
            xs[v] = stg + s * SP + n;
            ps[v] = f.spk + o;
            pm[v] = f.mem + o;
            pb[v] = f.bits ? f.bits + (o >> 3) : nullptr;
          }
          const int xstep = f.BS * SP;
          for (int ts = 0; ts < f.T; ++ts) {
#pragma unroll
            for (int v = 0; v < kScanLanes; ++v) {
              if (v >= nv) break;  // uniform: the whole group is past the tile
              const float x = *xs[v];
              xs[v] += xstep;
              float idummy = 0.0f;
              fwd_step<false, RESET, 0>(f.reset, beta[v], thr[v], 0.0f, x, u[v], z[v], idummy);
              const bool zz = ok[v] && z[v];
              if (ok[v]) {
                *ps[v] = __float2bfloat16_rn(zz ? 1.0f : 0.0f);
                *pm[v] = __float2bfloat16_rn(u[v]);
              }
              ps[v] += RN;
              pm[v] += RN;
              if (f.bits) {
                // 8 consecutive threads hold 8 consecutive lanes of one row (BN
                // and N are multiples of 8): one byte of the step's bit row
                const uint32_t m = __ballot_sync(0xffffffffu, zz);
                if ((lid & 7) == 0 && ok[v]) *pb[v] = (unsigned char)((m >> lid) & 0xFFu);
                pb[v] += f.bits_row;
              }
            }
          }
        }
      }
      epi_barrier();  // the staged rows are consumed before the next tile's copy
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, TCOLS);
  }
}

template <int BN, int RESET, bool BWD = false, int SG = 0>
cudaError_t launch_fused(const CUtensorMap& ta, const CUtensorMap& tb, const FusedArgs& f,
                         cudaStream_t st) {
  const void* k = (const void*)gemm_leaky_tcgen05<BN, RESET, BWD, SG>;
  const cudaError_t attr = ensure_smem(k, fused_smem_bytes<BN>());
  if (attr != cudaSuccess) return attr;
  int dev = 0, sms = 152, per_sm = 1;
  if (cudaGetDevice(&dev) == cudaSuccess) cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  // persistent CTAs: as many as fit at once (one CTA's scan overlaps the
  // other's main loop when two fit)
  if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, k, kFusedThreads, fused_smem_bytes<BN>()) !=
          cudaSuccess || per_sm < 1)
    per_sm = 1;
  if (fused_smem_bytes<BN>() * 2 <= 220 * 1024) per_sm = per_sm < 2 ? 2 : per_sm;  // fits twice
  const int64_t slots = (int64_t)sms * (per_sm > 2 ? 2 : per_sm);
  const int64_t tiles = (int64_t)((f.N + BN - 1) / BN) * ((f.R + f.BS - 1) / f.BS);
  const unsigned grid = (unsigned)(tiles < slots ? tiles : slots);
  return launch_pdl(gemm_leaky_tcgen05<BN, RESET, BWD, SG>, dim3(grid), dim3(kFusedThreads),
                    fused_smem_bytes<BN>(), st, ta, tb, f);
}

template <int BN, int SG>
cudaError_t launch_fused_bwd_reset(const CUtensorMap& ta, const CUtensorMap& tb, const FusedArgs& f,
                                   cudaStream_t st) {
  switch (f.reset) {
    case RESET_SUBTRACT: return launch_fused<BN, RESET_SUBTRACT, true, SG>(ta, tb, f, st);
    case RESET_ZERO: return launch_fused<BN, RESET_ZERO, true, SG>(ta, tb, f, st);
    default: return launch_fused<BN, RESET_NONE, true, SG>(ta, tb, f, st);
  }
}

template <int BN>
cudaError_t launch_fused_bwd(const CUtensorMap& ta, const CUtensorMap& tb, const FusedArgs& f,
                             cudaStream_t st) {
  return f.sa.sg == SG_FAST_SIGMOID ? launch_fused_bwd_reset<BN, SG_FAST_SIGMOID>(ta, tb, f, st)
                                    : launch_fused_bwd_reset<BN, SG_ATAN>(ta, tb, f, st);
}

template <int BN>
cudaError_t launch_fused_reset(const CUtensorMap& ta, const CUtensorMap& tb, const FusedArgs& f,
                               cudaStream_t st) {
  switch (f.reset) {
    case RESET_SUBTRACT: return launch_fused<BN, RESET_SUBTRACT>(ta, tb, f, st);
    case RESET_ZERO: return launch_fused<BN, RESET_ZERO>(ta, tb, f, st);
    default: return launch_fused<BN, RESET_NONE>(ta, tb, f, st);
  }
}

bool al16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

}  // namespace
}  // namespace gemm
}  // namespace snn

using namespace snn::gemm;

extern "C" snn_status_t snn_dense_leaky_fwd(const snn_scan_desc* d, int64_t P, int64_t K,
                                            const void* X, const void* W, const float* beta,
                                            const float* thr, void* spk, void* mem, float* ckpt,
                                            void* ws, size_t ws_bytes, snn_stream_t stream) {
  if (!d || P < 1 || K < 0) return SNN_ERR_INVALID_ARG;
  if (d->T < 1 || d->B < 1 || d->N < 1 || d->N % P != 0) return SNN_ERR_INVALID_ARG;
  if (d->reserved0 != 0 || d->reserved1 != 0) return SNN_ERR_INVALID_ARG;
  if (d->reset < SNN_RESET_SUBTRACT || d->reset > SNN_RESET_NONE) return SNN_ERR_INVALID_ARG;
  const int64_t Nout = d->N / P, R = d->B * P;
  if (d->io_dtype != SNN_BF16 || d->save != SNN_SAVE_MEM) return SNN_ERR_UNSUPPORTED;
  if (d->T > 128 || K % 8 != 0 || K == 0 || Nout % 8 != 0) return SNN_ERR_UNSUPPORTED;
  if (R > INT_MAX / 2 || K > INT_MAX / 2 || Nout > INT_MAX / 2 || d->T * R * Nout > (int64_t)1 << 46)
    return SNN_ERR_INVALID_ARG;
  // parameters: one value, or one per output column (per neuron of a dense
  // layer, per channel of a channel-last convolution)
  auto col_mode = [&](int32_t mode, int* col) {
    if (mode == SNN_P_SCALAR) { *col = 0; return true; }
    if (mode == SNN_P_PER_NEURON && P == 1) { *col = 1; return true; }
    if (mode == SNN_P_PER_CHANNEL && d->C == Nout && d->HW == 1) { *col = 1; return true; }
    return false;
  };
  int beta_col = 0, thr_col = 0;
  if (!col_mode(d->beta_mode, &beta_col) || !col_mode(d->thr_mode, &thr_col)) return SNN_ERR_UNSUPPORTED;
  if (!X || !W || !beta || !thr || !spk || !mem) return SNN_ERR_INVALID_ARG;
  if (!al16(X) || !al16(W) || !al16(spk) || !al16(mem) || (ckpt && !al16(ckpt)) || !al16(ws))
    return SNN_ERR_ALIGNMENT;
  if (!ws || ws_bytes < 256) return SNN_ERR_WORKSPACE;
  FusedArgs f{};
  f.T = (int)d->T;
  f.R = (int)R;
  f.K = (int)K;
  f.N = (int)Nout;
  f.BS = (int)(128 / d->T);
  f.reset = d->reset;
  f.beta_col = beta_col;
  f.thr_col = thr_col;
  f.beta = beta;
  f.thr = thr;
  f.spk = static_cast<__nv_bfloat16*>(spk);
  f.mem = static_cast<__nv_bfloat16*>(mem);
  f.bits = reinterpret_cast<unsigned char*>(ckpt);
  f.bits_row = ((d->B * d->N + 7) / 8 + 15) / 16 * 16;
  f.status = static_cast<int*>(ws);
  f.wait_ns = d->wait_limit_ns > 0 ? (uint64_t)d->wait_limit_ns : kDefaultWaitNs;
  // the widest tile the output needs, 64 rather than 128 when 128-wide tiles
  // would leave SMs without a second tile
  int bn = Nout <= 16 ? 16 : Nout <= 32 ? 32 : Nout <= 64 ? 64 : 128;
  if (bn == 128) {
    int dev = 0, sms = 152;
    if (cudaGetDevice(&dev) == cudaSuccess) cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    const int64_t tiles128 = ((Nout + 127) / 128) * ((R + f.BS - 1) / f.BS);
    if (tiles128 < 2 * (int64_t)sms) bn = 64;
  }
  CUtensorMap ta, tb;
  if (!make_map_3d(&ta, X, d->T, R, K, f.BS, (int)d->T) || !make_map(&tb, W, Nout, K, bn))
    return SNN_ERR_UNSUPPORTED;
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  cudaError_t e;
  switch (bn) {
    case 16: e = launch_fused_reset<16>(ta, tb, f, st); break;
    case 32: e = launch_fused_reset<32>(ta, tb, f, st); break;
    case 64: e = launch_fused_reset<64>(ta, tb, f, st); break;
    default: e = launch_fused_reset<128>(ta, tb, f, st);
  }
  return e == cudaSuccess ? SNN_OK : SNN_ERR_CUDA;
}

extern "C" snn_status_t snn_dense_leaky_bwd(const snn_scan_desc* d, int64_t K, const void* dI_up,
                                            const void* W, const float* beta, const float* thr,
                                            const void* mem, const void* spk, const float* ckpt,
                                            void* grad_I, void* ws, size_t ws_bytes,
                                            snn_stream_t stream) {
  if (!d || K < 0) return SNN_ERR_INVALID_ARG;
  if (d->T < 1 || d->B < 1 || d->N < 1 || d->reserved0 != 0 || d->reserved1 != 0)
    return SNN_ERR_INVALID_ARG;
  if (d->reset < SNN_RESET_SUBTRACT || d->reset > SNN_RESET_NONE) return SNN_ERR_INVALID_ARG;
  if (d->surrogate != SNN_SG_FAST_SIGMOID && d->surrogate != SNN_SG_ATAN) return SNN_ERR_INVALID_ARG;
  if (!(d->sg_param > 0.0f)) return SNN_ERR_INVALID_ARG;
  if (d->io_dtype != SNN_BF16 || d->save != SNN_SAVE_MEM) return SNN_ERR_UNSUPPORTED;
  if (d->T > 128 || K % 8 != 0 || K == 0 || d->N % 8 != 0) return SNN_ERR_UNSUPPORTED;
  if (d->B > INT_MAX / 2 || K > INT_MAX / 2 || d->N > INT_MAX / 2 || d->T * d->B * d->N > ((int64_t)1 << 46))
    return SNN_ERR_INVALID_ARG;
  auto col_mode = [&](int32_t mode, int* col) {
    if (mode == SNN_P_SCALAR) { *col = 0; return true; }
    if (mode == SNN_P_PER_NEURON) { *col = 1; return true; }
    return false;
  };
  int beta_col = 0, thr_col = 0;
  if (!col_mode(d->beta_mode, &beta_col) || !col_mode(d->thr_mode, &thr_col)) return SNN_ERR_UNSUPPORTED;
  if (!dI_up || !W || !beta || !thr || !mem || !grad_I || (!ckpt && !spk)) return SNN_ERR_INVALID_ARG;
  if (!al16(dI_up) || !al16(W) || !al16(mem) || !al16(grad_I) || (spk && !al16(spk)) ||
      (ckpt && !al16(ckpt)) || !al16(ws))
    return SNN_ERR_ALIGNMENT;
  if (!ws || ws_bytes < 256) return SNN_ERR_WORKSPACE;
  FusedArgs f{};
  f.T = (int)d->T;
  f.R = (int)d->B;
  f.K = (int)K;
  f.N = (int)d->N;
  f.BS = (int)(128 / d->T);
  f.reset = d->reset;
  f.beta_col = beta_col;
  f.thr_col = thr_col;
  f.beta = beta;
  f.thr = thr;
  f.bits_row = ((d->B * d->N + 7) / 8 + 15) / 16 * 16;
  f.status = static_cast<int*>(ws);
  f.wait_ns = d->wait_limit_ns > 0 ? (uint64_t)d->wait_limit_ns : kDefaultWaitNs;
  f.mem_in = static_cast<const __nv_bfloat16*>(mem);
  f.bits_in = reinterpret_cast<const unsigned char*>(ckpt);
  f.spk_in = static_cast<const __nv_bfloat16*>(spk);
  f.gI = static_cast<__nv_bfloat16*>(grad_I);
  f.sa.reset = d->reset;
  f.sa.detach = d->detach_reset != 0;
  f.sa.sg = d->surrogate;
  f.sa.rec = 0;
  if (d->surrogate == SNN_SG_FAST_SIGMOID) {
    f.sa.sg_a = d->sg_param;
    f.sa.sg_b = 0.0f;
  } else {  // the same constants the scan kernels take
    f.sa.sg_a = (float)(0.5 * (double)d->sg_param);
    f.sa.sg_b = (float)(3.14159265358979323846 * 0.5 * (double)d->sg_param);
  }
  // 128-wide tiles unless 64-wide ones are needed to give the SMs a second tile
  int bn = 128;
  {
    int dev = 0, sms = 152;
    if (cudaGetDevice(&dev) == cudaSuccess) cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    const int64_t tiles128 = ((d->N + 127) / 128) * ((d->B + f.BS - 1) / f.BS);
    if (d->N <= 64 || tiles128 < 2 * (int64_t)sms) bn = 64;
  }
  CUtensorMap ta, tb;
  if (!make_map_3d(&ta, dI_up, d->T, d->B, K, f.BS, (int)d->T) || !make_map(&tb, W, K, d->N, 64))
    return SNN_ERR_UNSUPPORTED;
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  const cudaError_t e = bn == 64 ? launch_fused_bwd<64>(ta, tb, f, st) : launch_fused_bwd<128>(ta, tb, f, st);
  return e == cudaSuccess ? SNN_OK : SNN_ERR_CUDA;
}
