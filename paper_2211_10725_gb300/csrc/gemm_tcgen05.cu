// Dense-layer input current on the 5th-generation tensor cores: the synaptic
// operation w.x of the paper's Fig. 3 batched over all T*B rows,
//   D[M, N] = A[M, K] * B[N, K]^T,   A, B bf16 row-major (K contiguous),
// fp32 accumulation in tensor memory, fp32 or bf16 output.
//
// Persistent CTAs (one per SM) take 128 x BN tiles (BN up to 256) in turn.  Warp 0 (one
// thread) streams 128x64 and BNx64 operand tiles into a shared-memory ring
// with TMA (128-byte swizzle), 8, 6 or 4 stages deep for BN = 64, 128, 256
// (as deep as fits beside the output staging); warp 1 allocates two TMEM
// accumulators and one thread issues tcgen05.mma (M=128, N=BN, K=16 per
// instruction) as stages land, freeing each stage through tcgen05.commit;
// warps 2-5 read a finished accumulator back with tcgen05.ld (each warp its
// 32-lane quarter) and store it while the next tile accumulates in the
// other buffer.  Every wait
// is bounded; a kernel that gives up records SNN_ERR_TIMEOUT and still
// drains its copies and frees its TMEM.
//
// Either operand may instead be stored MN-major (its M or N index
// contiguous, K the row index): the backward products dX = dI*W (W read
// MN-major) and dW = dI^T*X (dI and X read MN-major) then run on the stored
// matrices without transposed copies.  An MN-major tile is loaded as
// 64-element-wide TMA boxes (64 MN x 64 K, 128-byte swizzle) and described
// to the tensor core as atoms of 8 K-rows of 128 bytes: 1024 bytes apart
// along K, one box (8 KB) apart along MN.
//
// Output: with 16-byte output rows each epilogue warp stages its 32 rows
// of a 128-byte-wide column chunk in shared memory (128-byte swizzle, two
// buffers per warp) and one lane writes the chunk with a TMA tensor store,
// so every warp write is whole 128-byte lines; otherwise the threads store
// their rows directly.
//
// Split K: a product whose few output tiles each sum a long K (the weight
// gradient of a convolution sums over every patch row) runs as tiles x S
// work items, item (tile, s) summing k-blocks [s*nk/S, (s+1)*nk/S) into
// partial output s; a second kernel adds the S partials in split order, so
// the result does not depend on which CTA ran which item.  Weight gradients
// of wide layers use 128 x 256 tiles (four 64-column MN-major B boxes) and
// splits, which cuts the re-reads of dI across output columns.
#include <cuda.h>
#include <cudaTypedefs.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include <climits>
#include <cstdint>
#include <cstring>
#include <mutex>

#include "scan_host.cuh"
#include "snn.h"
#include "tcgen05.cuh"

namespace snn {
namespace gemm {

struct GemmArgs {
  int M, N, K;
  void* D;
  int64_t ldd;  // row stride of D in elements
  int* status;
  uint64_t wait_ns;
  int ksplit;            // K splits per tile (1: D is the result)
  int64_t split_stride;  // elements between the partial outputs of two splits
};

// ---------------------------------------------------------------------------
// Kernel: persistent, work items blockIdx.x, blockIdx.x + gridDim.x, ...;
// item i is split i % S of tile i / S, tiles in row-major order (N tiles
// fastest).  The operand ring runs on across
// tiles; the accumulator alternates between two TMEM buffers so that the
// epilogue of one tile overlaps the main loop of the next.
// ---------------------------------------------------------------------------

template <int BN, bool OUT_BF16, bool A_MN = false, bool B_MN = false, bool TMA_OUT = false>
__global__ void __launch_bounds__(kThreads, kCtasPerSm)
    gemm_tn_tcgen05(const __grid_constant__ CUtensorMap ta, const __grid_constant__ CUtensorMap tb,
                    const __grid_constant__ CUtensorMap td, const GemmArgs g) {
  static_assert(BN % 16 == 0 && BN >= 16 && BN <= 256, "UMMA N for M=128, two accumulators");
  static_assert(!B_MN || BN % 64 == 0, "an MN-major B tile is whole 64-wide boxes");
  constexpr int OUT_CW = OUT_BF16 ? 64 : 32;  // columns of one 128-byte output chunk
  static_assert(!TMA_OUT || BN % OUT_CW == 0, "the tile is whole output chunks");
  constexpr int A_BYTES = BM * BK * 2;
  constexpr int B_BYTES = BN * BK * 2;
  constexpr uint32_t TCOLS = tmem_cols<BN>();
  constexpr int kEpiWarps = 4;
  constexpr int kStages = gemm_stages<BN>();
  static_assert(smem_bytes<BN, TMA_OUT>() <= 227 * 1024, "the ring and staging fit one CTA");
  extern __shared__ unsigned char smem_raw[];
  unsigned char* smem =
      reinterpret_cast<unsigned char*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  unsigned char* sA = smem;
  unsigned char* sB = smem + kStages * A_BYTES;
  unsigned char* sOut = sB + kStages * B_BYTES;  // output staging (TMA_OUT), 1024-aligned
  uint64_t* full = reinterpret_cast<uint64_t*>(sOut + (TMA_OUT ? kOutStaging : 0));
  uint64_t* empty = full + kStages;
  uint64_t* acc_full = empty + kStages;  // [2] MMA -> epilogue
  uint64_t* acc_empty = acc_full + 2;    // [2] epilogue -> MMA
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(acc_empty + 2);
  const int warp = threadIdx.x >> 5, lid = threadIdx.x & 31;
  const int nk = (g.K + BK - 1) / BK;
  const int tiles_n = (g.N + BN - 1) / BN;
  const int S = g.ksplit;
  const int items = tiles_n * ((g.M + BM - 1) / BM) * S;  // (tile, split), split fastest

  if (threadIdx.x == 0) {
    for (int s = 0; s < kStages; ++s) {
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
  grid_dep_wait();  // the previous kernel on the stream is complete

  if (warp == 0) {
    if (lid == 0) {
      int64_t n_issued = 0;  // k-blocks issued over all tiles: ring position
      bool ok = true;
      for (int it = blockIdx.x; it < items && ok; it += gridDim.x) {
        const int t = it / S, sp = it - t * S;
        const int m0 = (t / tiles_n) * BM, n0 = (t % tiles_n) * BN;
        const int kb1 = (int)((int64_t)nk * (sp + 1) / S);
        for (int kb = (int)((int64_t)nk * sp / S); kb < kb1; ++kb, ++n_issued) {
          const int s = (int)(n_issued % kStages);
          if (n_issued >= kStages &&
              !mbar_wait_poll(&empty[s], (uint32_t)(((n_issued / kStages) - 1) & 1), g.wait_ns)) {
            record_status(g.status, kStatusTimeout);
            ok = false;
            break;
          }
          mbar_arrive_expect_tx(&full[s], A_BYTES + B_BYTES);
          if (A_MN) {
#pragma unroll
            for (int j = 0; j < BM / 64; ++j)
              tma_load_2d(sA + s * A_BYTES + j * kMnBoxBytes, &ta, m0 + 64 * j, kb * BK, &full[s]);
          } else {
            tma_load_2d(sA + s * A_BYTES, &ta, kb * BK, m0, &full[s]);
          }
          if (B_MN) {
#pragma unroll
            for (int j = 0; j < BN / 64; ++j)
              tma_load_2d(sB + s * B_BYTES + j * kMnBoxBytes, &tb, n0 + 64 * j, kb * BK, &full[s]);
          } else {
            tma_load_2d(sB + s * B_BYTES, &tb, kb * BK, n0, &full[s]);
          }
        }
      }
      // every copy this thread issued has landed before the CTA may exit
      for (int64_t j = n_issued > kStages ? n_issued - kStages : 0; j < n_issued; ++j)
        mbar_wait_bounded(&full[j % kStages], (uint32_t)((j / kStages) & 1), kDrainWaitNs);
    }
  } else if (warp == 1) {
    if (lid == 0) {
      constexpr uint32_t idesc = idesc_bf16(BM, BN, A_MN, B_MN);
      // 16 more along K: 32 bytes inside a K-major row, or 16 rows (2048
      // bytes) of an MN-major tile; the descriptor holds the address >> 4
      constexpr uint64_t stepA = A_MN ? 2048 >> 4 : 32 >> 4;
      constexpr uint64_t stepB = B_MN ? 2048 >> 4 : 32 >> 4;
      int64_t n_used = 0;  // k-blocks consumed over all tiles
      bool ok = true;
      int i = 0;  // this CTA's tile count
      for (int it = blockIdx.x; it < items && ok; it += gridDim.x, ++i) {
        const int sp = it % S;
        const int kb0 = (int)((int64_t)nk * sp / S), kb1 = (int)((int64_t)nk * (sp + 1) / S);
        const int b = i & 1;
        // the epilogue has drained this accumulator (its use two tiles ago)
        if (i >= 2 && !mbar_wait_poll(&acc_empty[b], (uint32_t)(((i >> 1) - 1) & 1), g.wait_ns)) {
          record_status(g.status, kStatusTimeout);
          break;
        }
        tc_fence_after();
        const uint32_t acc = tmem + (uint32_t)(b * BN);
        for (int kb = kb0; kb < kb1; ++kb, ++n_used) {
          const int s = (int)(n_used % kStages);
          if (!mbar_wait_poll(&full[s], (uint32_t)((n_used / kStages) & 1), g.wait_ns)) {
            record_status(g.status, kStatusTimeout);
            ok = false;
            break;
          }
          tc_fence_after();
          const uint64_t da = A_MN ? sdesc_sw128_mn(sA + s * A_BYTES) : sdesc_sw128(sA + s * A_BYTES);
          const uint64_t db = B_MN ? sdesc_sw128_mn(sB + s * B_BYTES) : sdesc_sw128(sB + s * B_BYTES);
#pragma unroll
          for (int kk = 0; kk < BK / 16; ++kk)
            tc_mma(acc, da + stepA * kk, db + stepB * kk, idesc, (kb != kb0 || kk != 0) ? 1u : 0u);
          tc_commit(&empty[s]);  // the stage is free once these MMAs are done
        }
        if (ok) tc_commit(&acc_full[b]);  // the tile's accumulator is final
      }
    }
  } else {
    // epilogue: warp w reads TMEM lanes 32*(w%4) .. +32, i.e. tile rows
    const int q = warp & 3;
    unsigned char* stage_out = sOut + q * 2 * kOutChunkBytes;
    int nchunk = 0;  // chunks this warp has staged (buffer parity)
    int i = 0;
    for (int it = blockIdx.x; it < items; it += gridDim.x, ++i) {
      const int t = it / S, sp = it - t * S;
      const int b = i & 1;
      if (!warp_wait_uniform(&acc_full[b], (uint32_t)((i >> 1) & 1), g.wait_ns)) {
        if (lid == 0) record_status(g.status, kStatusTimeout);
        break;
      }
      tc_fence_after();
      const int m0 = (t / tiles_n) * BM, n0 = (t % tiles_n) * BN;
      const int row = m0 + q * 32 + lid;
      void* const Dout = OUT_BF16 ? (void*)(static_cast<__nv_bfloat16*>(g.D) + sp * g.split_stride)
                                  : (void*)(static_cast<float*>(g.D) + sp * g.split_stride);
      const uint32_t acc = tmem + ((uint32_t)(q * 32) << 16) + (uint32_t)(b * BN);
      if constexpr (TMA_OUT) {
        // 128-byte column chunks: TMEM -> registers -> swizzled staging ->
        // TMA store (rows and columns past M and N are clipped by the map)
#pragma unroll 1
        for (int c = 0; c < BN && n0 + c < g.N; c += OUT_CW) {
          unsigned char* buf = stage_out + (nchunk & 1) * kOutChunkBytes;
          if (lid == 0) bulk_wait_read_all_but_one();  // this buffer's last store has read it
          __syncwarp();
          unsigned char* rowp = buf + lid * 128;
#pragma unroll
          for (int cc = 0; cc < OUT_CW; cc += 16) {
            uint32_t r[16];
            tmem_ld16(acc + (uint32_t)(c + cc), r);
            if (OUT_BF16) {
              uint32_t w[8];
#pragma unroll
              for (int j = 0; j < 8; ++j) {
                __nv_bfloat162 h = __floats2bfloat162_rn(__uint_as_float(r[2 * j]), __uint_as_float(r[2 * j + 1]));
                w[j] = *reinterpret_cast<uint32_t*>(&h);
              }
              const int j0 = cc / 8;  // 16-byte chunk index of column cc within the row
              *reinterpret_cast<uint4*>(rowp + (((j0) ^ (lid & 7)) << 4)) = make_uint4(w[0], w[1], w[2], w[3]);
              *reinterpret_cast<uint4*>(rowp + (((j0 + 1) ^ (lid & 7)) << 4)) = make_uint4(w[4], w[5], w[6], w[7]);
            } else {
              const int j0 = cc / 4;
#pragma unroll
              for (int j = 0; j < 4; ++j)
                *reinterpret_cast<uint4*>(rowp + (((j0 + j) ^ (lid & 7)) << 4)) =
                    make_uint4(r[4 * j], r[4 * j + 1], r[4 * j + 2], r[4 * j + 3]);
            }
          }
          fence_async_smem();
          __syncwarp();
          if (lid == 0) {
            tma_store_3d(&td, buf, n0 + c, m0 + q * 32, sp);
            bulk_commit();
          }
          ++nchunk;
        }
      } else {
#pragma unroll 1
      for (int c = 0; c < BN; c += 16) {
        uint32_t r[16];
        tmem_ld16(acc + (uint32_t)c, r);
        const int col = n0 + c;
        if (row < g.M && col < g.N) {
          if (OUT_BF16) {
            __nv_bfloat16* d = static_cast<__nv_bfloat16*>(Dout) + (int64_t)row * g.ldd + col;
            if (col + 16 <= g.N && (((int64_t)row * g.ldd + col) & 7) == 0) {
              uint4 v[2];
              uint32_t* w = reinterpret_cast<uint32_t*>(v);
#pragma unroll
              for (int j = 0; j < 8; ++j) {
                __nv_bfloat162 h = __floats2bfloat162_rn(__uint_as_float(r[2 * j]), __uint_as_float(r[2 * j + 1]));
                w[j] = *reinterpret_cast<uint32_t*>(&h);
              }
              reinterpret_cast<uint4*>(d)[0] = v[0];
              reinterpret_cast<uint4*>(d)[1] = v[1];
            } else {
              for (int j = 0; j < 16 && col + j < g.N; ++j) d[j] = __float2bfloat16_rn(__uint_as_float(r[j]));
            }
          } else {
            float* d = static_cast<float*>(Dout) + (int64_t)row * g.ldd + col;
            if (col + 16 <= g.N && (((int64_t)row * g.ldd + col) & 3) == 0) {
#pragma unroll
              for (int j = 0; j < 4; ++j)
                reinterpret_cast<float4*>(d)[j] =
                    make_float4(__uint_as_float(r[4 * j]), __uint_as_float(r[4 * j + 1]),
                                __uint_as_float(r[4 * j + 2]), __uint_as_float(r[4 * j + 3]));
            } else {
              for (int j = 0; j < 16 && col + j < g.N; ++j) d[j] = __uint_as_float(r[j]);
            }
          }
        }
      }
      }
      // this warp's reads of the accumulator are done: hand it back
      tc_fence_before();
      __syncwarp();
      if (lid == 0) mbar_arrive(&acc_empty[b]);
    }
    if (TMA_OUT && lid == 0) bulk_wait_all();  // the staged chunks are written out
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, TCOLS);
  }
}

// ---------------------------------------------------------------------------
// Host side
// ---------------------------------------------------------------------------

template <int BN, bool OUT_BF16, bool A_MN, bool B_MN, bool TMA_OUT>
cudaError_t launch_bn(const CUtensorMap& ta, const CUtensorMap& tb, const CUtensorMap& td,
                      const GemmArgs& g, cudaStream_t st) {
  const void* k = (const void*)gemm_tn_tcgen05<BN, OUT_BF16, A_MN, B_MN, TMA_OUT>;
  const cudaError_t attr = ensure_smem(k, smem_bytes<BN, TMA_OUT>());  // once per device
  if (attr != cudaSuccess) return attr;
  int dev = 0, sms = 152;
  if (cudaGetDevice(&dev) == cudaSuccess)
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  const int64_t items = (int64_t)((g.N + BN - 1) / BN) * ((g.M + BM - 1) / BM) * g.ksplit;
  const int64_t slots = (int64_t)sms * kCtasPerSm;
  const unsigned grid = (unsigned)(items < slots ? items : slots);  // persistent CTAs
  return launch_pdl(gemm_tn_tcgen05<BN, OUT_BF16, A_MN, B_MN, TMA_OUT>, dim3(grid),
                    dim3(kThreads), smem_bytes<BN, TMA_OUT>(), st, ta, tb, td, g);
}

// The TMA-store epilogue when the output rows are 16-byte multiples and
// the tile is whole 128-byte chunks; else direct stores.
template <int BN, bool OUT_BF16, bool A_MN, bool B_MN>
cudaError_t launch_out(const CUtensorMap& ta, const CUtensorMap& tb, const GemmArgs& g,
                       cudaStream_t st) {
  constexpr int cw = OUT_BF16 ? 64 : 32;
  CUtensorMap td;
  if constexpr (BN % cw == 0) {
    const int64_t es = OUT_BF16 ? 2 : 4;
    if (((int64_t)g.N * es) % 16 == 0 && (reinterpret_cast<uintptr_t>(g.D) & 15u) == 0 &&
        make_out_map(&td, g.D, g.ksplit, g.M, g.N, OUT_BF16))
      return launch_bn<BN, OUT_BF16, A_MN, B_MN, true>(ta, tb, td, g, st);
  }
  memset(&td, 0, sizeof(td));
  return launch_bn<BN, OUT_BF16, A_MN, B_MN, false>(ta, tb, td, g, st);
}

// D[M, N] = A[M, K] * B[N, K]^T.  A is stored [M, K] row-major (K-major) or,
// with A_MN, [K, M] row-major; B likewise [N, K] or, with B_MN, [K, N].
// N tile: the widest the output needs (64, 128 or 192 for an MN-major B),
// and 64 rather than 128 when 128-wide tiles would leave most SMs idle.
template <bool OUT_BF16, bool A_MN = false, bool B_MN = false>
cudaError_t gemm_tn(const void* A, const void* B, void* D, int M, int N, int K, int* status,
                    cudaStream_t st, int ksplit = 1, int bn_force = 0) {
  // a 128 x 256 tile keeps the tensor core busier per instruction (about
  // 1.6x the rate of 128 x 128 at large K); below K = 512 the per-tile
  // fixed costs dominate and the narrower tile's parallelism wins
  int bn = (!B_MN && N > 128 && K >= 512) ? 256 : 128;
  if (bn_force > 0) bn = bn_force;
  else if (N <= 16 && !B_MN) bn = 16;
  else if (N <= 32 && !B_MN) bn = 32;
  else if (N <= 64) bn = 64;
  // an MN-major B wider than two 128-column tiles: 192-wide tiles when
  // they need fewer tiles (each re-reads its A rows once)
  else if (B_MN && N > 256 && (N + 191) / 192 < (N + 127) / 128) bn = 192;
  else {
    int dev = 0, sms = 152;
    if (cudaGetDevice(&dev) == cudaSuccess)
      cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    const int64_t tiles128 = (int64_t)((N + 127) / 128) * ((M + BM - 1) / BM);
    if (tiles128 < (int64_t)sms * kCtasPerSm) bn = 64;
  }
  CUtensorMap ta, tb;
  const bool okA = A_MN ? make_map(&ta, A, K, M, 64) : make_map(&ta, A, M, K, BM);
  const bool okB = B_MN ? make_map(&tb, B, K, N, 64) : make_map(&tb, B, N, K, bn);
  if (!okA || !okB) return cudaErrorInvalidValue;
  GemmArgs g{M, N, K, D, (int64_t)N, status, kDefaultWaitNs, ksplit, (int64_t)M * N};
  if constexpr (B_MN) {
    if (bn == 64) return launch_out<64, OUT_BF16, A_MN, B_MN>(ta, tb, g, st);
    if (bn == 256) return launch_out<256, OUT_BF16, A_MN, B_MN>(ta, tb, g, st);
    if (bn == 192) return launch_out<192, OUT_BF16, A_MN, B_MN>(ta, tb, g, st);
    return launch_out<128, OUT_BF16, A_MN, B_MN>(ta, tb, g, st);
  } else {
    switch (bn) {
      case 256: return launch_out<256, OUT_BF16, A_MN, B_MN>(ta, tb, g, st);
      case 16: return launch_out<16, OUT_BF16, A_MN, B_MN>(ta, tb, g, st);
      case 32: return launch_out<32, OUT_BF16, A_MN, B_MN>(ta, tb, g, st);
      case 64: return launch_out<64, OUT_BF16, A_MN, B_MN>(ta, tb, g, st);
      default: return launch_out<128, OUT_BF16, A_MN, B_MN>(ta, tb, g, st);
    }
  }
}

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }
size_t round256(size_t b) { return (b + 255) & ~size_t(255); }

// K splits of the weight-gradient product dW[N, K] = dI^T X (reduction over
// the M rows), from the shapes alone so that a shape always sums in the same
// order: enough (tile, split) items to give each of about one GPU's worth of
// SMs (kSplitSlots) one, with at least kMinSplitKBlocks k-blocks per split.
// 128 x 256 tiles for K >= 256 inputs when the splits still give the SMs
// work (always for a wide layer, N >= 256 neurons and K >= 512; for a
// narrow one, such as a convolution's 64 channels over 304 patch columns,
// when the reduction is long enough for at least 3/4 of kSplitSlots items):
// dI is re-read once per 256 columns instead of once per 64.  Otherwise
// the GEMM's own tile choice, split to fill the SMs.
constexpr int64_t kSplitSlots = 152;
constexpr int64_t kMinSplitKBlocks = 8;
struct DwPlan {
  int bn;  // 0: the GEMM's own choice
  int S;
};
DwPlan dw_plan(int64_t M, int64_t K, int64_t N) {
  const int64_t nk = (M + BK - 1) / BK;
  auto splits = [&](int64_t tiles) {
    int64_t s = kSplitSlots / (tiles > 0 ? tiles : 1);
    if (s > nk / kMinSplitKBlocks) s = nk / kMinSplitKBlocks;
    return s < 1 ? 1 : (int)s;
  };
  if (K >= 256) {
    const int64_t tiles = ((N + BM - 1) / BM) * ((K + 255) / 256);
    const int S = splits(tiles);
    if (S >= 2 && ((N >= 256 && K >= 512) || tiles * S >= kSplitSlots * 3 / 4)) return DwPlan{256, S};
  }
  return DwPlan{0, splits(((N + BM - 1) / BM) * ((K + 63) / 64))};
}
int dw_splits(int64_t M, int64_t K, int64_t N) { return dw_plan(M, K, N).S; }

// out[i] = sum over s = 0 .. S-1 of part[s * n + i], in split order.
__global__ void __launch_bounds__(256) sum_splits(const float4* __restrict__ part,
                                                  float4* __restrict__ out, int64_t n4, int S) {
  grid_dep_wait();
  const int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= n4) return;
  float4 a = part[i];
  for (int s = 1; s < S; ++s) {
    const float4 b = part[(int64_t)s * n4 + i];
    a.x += b.x;
    a.y += b.y;
    a.z += b.z;
    a.w += b.w;
  }
  out[i] = a;
}

snn_status_t check_dims(int64_t M, int64_t K, int64_t N) {
  if (M < 0 || K < 0 || N < 0) return SNN_ERR_INVALID_ARG;
  if (M > INT_MAX / 2 || K > INT_MAX / 2 || N > INT_MAX / 2) return SNN_ERR_INVALID_ARG;
  return SNN_OK;
}

}  // namespace gemm
}  // namespace snn

using namespace snn::gemm;

extern "C" {

size_t snn_dense_workspace_bytes(int64_t M, int64_t K, int64_t N) {
  if (check_dims(M, K, N) != SNN_OK) return 0;
  // the status word (the backward reads its operands in place), then the
  // split-K partials of dW when the weight gradient is split
  const int S = dw_splits(M, K, N);
  return 256 + (S > 1 ? round256((size_t)S * N * K * sizeof(float)) : 0);
}

snn_status_t snn_dense_layer_fwd(int64_t M, int64_t K, int64_t N, const void* X, const void* W,
                                 float* I, void* ws, size_t ws_bytes, snn_stream_t stream) {
  snn_status_t s = check_dims(M, K, N);
  if (s != SNN_OK) return s;
  if (K % 8 != 0) return SNN_ERR_UNSUPPORTED;  // TMA needs 16-byte row strides
  if ((M > 0 && N > 0) && (!X || !W || !I)) return SNN_ERR_INVALID_ARG;
  if (!aligned16(X) || !aligned16(W) || !aligned16(I) || !aligned16(ws)) return SNN_ERR_ALIGNMENT;
  if (!ws || ws_bytes < 256) return SNN_ERR_WORKSPACE;
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  if (M == 0 || N == 0) return SNN_OK;
  if (K == 0)
    return cudaMemsetAsync(I, 0, (size_t)M * N * sizeof(float), st) == cudaSuccess ? SNN_OK : SNN_ERR_CUDA;
  const cudaError_t e = gemm_tn<false>(X, W, I, (int)M, (int)N, (int)K, static_cast<int*>(ws), st);
  return e == cudaSuccess ? SNN_OK : (e == cudaErrorInvalidValue ? SNN_ERR_UNSUPPORTED : SNN_ERR_CUDA);
}

snn_status_t snn_dense_layer_bwd(int64_t M, int64_t K, int64_t N, const void* X, const void* W,
                                 const void* dI, void* dX, float* dW, void* ws, size_t ws_bytes,
                                 snn_stream_t stream) {
  snn_status_t s = check_dims(M, K, N);
  if (s != SNN_OK) return s;
  if (K % 8 != 0 || N % 8 != 0 || M % 8 != 0) return SNN_ERR_UNSUPPORTED;
  if (!dI || (!dX && !dW)) return SNN_ERR_INVALID_ARG;
  if ((dX && !W) || (dW && !X)) return SNN_ERR_INVALID_ARG;
  const void* ptrs[6] = {X, W, dI, dX, dW, ws};
  for (const void* p : ptrs)
    if (!aligned16(p)) return SNN_ERR_ALIGNMENT;
  if (!ws || ws_bytes < snn_dense_workspace_bytes(M, K, N)) return SNN_ERR_WORKSPACE;
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  int* status = static_cast<int*>(ws);
  cudaError_t e = cudaSuccess;
  if (dX && M > 0 && K > 0) {
    // dX[M, K] = dI[M, N] * W[N, K]: W is the MN-major B operand
    if (N == 0) e = cudaMemsetAsync(dX, 0, (size_t)M * K * 2, st);
    else e = gemm_tn<true, false, true>(dI, W, dX, (int)M, (int)K, (int)N, status, st);
    if (e != cudaSuccess) return e == cudaErrorInvalidValue ? SNN_ERR_UNSUPPORTED : SNN_ERR_CUDA;
  }
  if (dW && N > 0 && K > 0) {
    // dW[N, K] = dI[M, N]^T * X[M, K]: both operands MN-major (K = M here)
    const DwPlan plan = dw_plan(M, K, N);
    const int S = plan.S;
    if (M == 0) {
      e = cudaMemsetAsync(dW, 0, (size_t)N * K * sizeof(float), st);
    } else if (S == 1) {
      e = gemm_tn<false, true, true>(dI, X, dW, (int)N, (int)K, (int)M, status, st, 1, plan.bn);
    } else {
      float* part = reinterpret_cast<float*>(static_cast<unsigned char*>(ws) + 256);
      e = gemm_tn<false, true, true>(dI, X, part, (int)N, (int)K, (int)M, status, st, S, plan.bn);
      const int64_t n4 = N * K / 4;  // K is a multiple of 8
      if (e == cudaSuccess)
        e = snn::launch_pdl(sum_splits, dim3((unsigned)((n4 + 255) / 256)), dim3(256), 0, st,
                       reinterpret_cast<const float4*>(part), reinterpret_cast<float4*>(dW), n4, S);
    }
    if (e != cudaSuccess) return e == cudaErrorInvalidValue ? SNN_ERR_UNSUPPORTED : SNN_ERR_CUDA;
  }
  return SNN_OK;
}

}  // extern "C"
