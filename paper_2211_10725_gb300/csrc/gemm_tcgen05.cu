// Dense-layer input current on the 5th-generation tensor cores: the synaptic
// operation w.x of the paper's Fig. 3 batched over all T*B rows,
//   D[M, N] = A[M, K] * B[N, K]^T,   A, B bf16 row-major (K contiguous),
// fp32 accumulation in tensor memory, fp32 or bf16 output.
//
// Persistent CTAs (one per SM) take 128 x BN tiles (BN up to 256) in turn.  Warp 0 (one
// thread) streams 128x64 and BNx64 operand tiles into a 4-stage
// shared-memory ring with TMA (128-byte swizzle); warp 1 allocates two TMEM
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
// the result does not depend on which CTA ran which item.
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

namespace snn {
namespace gemm {

#ifndef SNN_GEMM_STAGES
#define SNN_GEMM_STAGES 4
#endif
#ifndef SNN_GEMM_CTAS_PER_SM
#define SNN_GEMM_CTAS_PER_SM 1
#endif
#ifndef SNN_GEMM_SLEEP_WAIT
#define SNN_GEMM_SLEEP_WAIT 0
#endif

constexpr int BM = 128;
constexpr int BK = 64;  // 64 bf16 = 128 bytes: one swizzle atom row
constexpr int kStages = SNN_GEMM_STAGES;
constexpr int kCtasPerSm = SNN_GEMM_CTAS_PER_SM;  // resident CTAs the tile size aims for
constexpr int kThreads = 192;
constexpr uint64_t kDefaultWaitNs = 2000000000ull;
constexpr uint64_t kDrainWaitNs = 1000000000ull;

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
// PTX wrappers: TMA, tcgen05
// ---------------------------------------------------------------------------

__device__ __forceinline__ void tma_load_2d(void* dst, const CUtensorMap* map, int x, int y,
                                            uint64_t* bar) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3}], [%4];" ::"r"(
          smem_u32(dst)),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(smem_u32(bar))
      : "memory");
}

__device__ __forceinline__ void tc_fence_before() {
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
}
__device__ __forceinline__ void tc_fence_after() {
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
}

// Shared-memory matrix descriptor of a K-major operand tile in the 128-byte
// swizzled layout TMA writes: rows of 128 bytes, 8-row (1024-byte) atoms.
__device__ __forceinline__ uint64_t sdesc_sw128(const void* tile) {
  const uint32_t addr = smem_u32(tile);
  uint64_t d = 0;
  d |= (uint64_t)((addr >> 4) & 0x3FFFu);      // start address
  d |= (uint64_t)(16u >> 4) << 16;              // leading byte offset (unused here)
  d |= (uint64_t)(1024u >> 4) << 32;            // stride byte offset: one 8-row atom
  d |= (uint64_t)1 << 46;                       // descriptor version
  d |= (uint64_t)2 << 61;                       // 128-byte swizzle
  return d;
}

// Descriptor of an MN-major operand tile: 64-element (128-byte) rows along
// MN for consecutive K; atoms of 8 K-rows (1024 bytes) repeat along K every
// 1024 bytes and along MN every 64x64 box (8192 bytes).
constexpr uint32_t kMnBoxBytes = 64 * BK * 2;
__device__ __forceinline__ uint64_t sdesc_sw128_mn(const void* tile) {
  const uint32_t addr = smem_u32(tile);
  uint64_t d = 0;
  d |= (uint64_t)((addr >> 4) & 0x3FFFu);      // start address
  d |= (uint64_t)(kMnBoxBytes >> 4) << 16;      // leading byte offset: next 64 along MN
  d |= (uint64_t)(1024u >> 4) << 32;            // stride byte offset: next 8 along K
  d |= (uint64_t)1 << 46;                       // descriptor version
  d |= (uint64_t)2 << 61;                       // 128-byte swizzle
  return d;
}

// Instruction descriptor: bf16 x bf16 -> fp32; each operand K-major or
// (a_mn / b_mn) MN-major.
__host__ __device__ constexpr uint32_t idesc_bf16(int m, int n, bool a_mn = false,
                                                  bool b_mn = false) {
  return (1u << 4)                         // D format: f32
         | (1u << 7)                       // A format: bf16
         | (1u << 10)                      // B format: bf16
         | ((a_mn ? 1u : 0u) << 15)        // A major-ness: MN
         | ((b_mn ? 1u : 0u) << 16)        // B major-ness: MN
         | ((uint32_t)(n >> 3) << 17)      // N / 8
         | ((uint32_t)(m >> 4) << 24);     // M / 16
}

__device__ __forceinline__ void tc_mma(uint32_t tmem_d, uint64_t adesc, uint64_t bdesc,
                                       uint32_t idesc, uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(tmem_d),
      "l"(adesc), "l"(bdesc), "r"(idesc), "r"(accumulate)
      : "memory");
}

// Arrive on `bar` once every tcgen05.mma this thread issued has completed.
__device__ __forceinline__ void tc_commit(uint64_t* bar) {
  asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(
                   smem_u32(bar))
               : "memory");
}

__device__ __forceinline__ void tmem_alloc(uint32_t* slot, uint32_t ncols) {
  asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(slot)),
               "r"(ncols)
               : "memory");
  asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
}

__device__ __forceinline__ void tmem_dealloc(uint32_t taddr, uint32_t ncols) {
  asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(taddr), "r"(ncols)
               : "memory");
}

// 32 lanes x 16 consecutive 32-bit columns of TMEM -> 16 registers per thread.
__device__ __forceinline__ void tmem_ld16(uint32_t taddr, uint32_t r[16]) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x16.b32 {%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, "
      "%12, %13, %14, %15}, [%16];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]),
        "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]),
        "=r"(r[14]), "=r"(r[15])
      : "r"(taddr));
  asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
}

// Bounded wait of the single producer / MMA thread on the critical path:
// polls without the suspend hint (a suspended thread can resume late), and
// reads the clock only every 64 polls.
__device__ __forceinline__ bool mbar_wait_poll(uint64_t* bar, uint32_t parity, uint64_t limit_ns) {
#if SNN_GEMM_SLEEP_WAIT
  return mbar_wait_bounded(bar, parity, limit_ns);
#else
  if (mbar_try_wait(bar, parity)) return true;
  const uint64_t t0 = globaltimer_ns();
  for (uint32_t i = 1;; ++i) {
    if (mbar_try_wait(bar, parity)) return true;
    if ((i & 63u) == 0 && globaltimer_ns() - t0 > limit_ns) return false;
  }
#endif
}

// Bounded wait taken by a whole warp; the give-up decision is warp-uniform.
__device__ __forceinline__ bool warp_wait_uniform(uint64_t* bar, uint32_t parity, uint64_t limit_ns) {
  bool done = mbar_try_wait(bar, parity);
  if (__all_sync(0xffffffffu, done)) return true;
  const uint64_t t0 = globaltimer_ns();
  while (true) {
    if (!done) done = mbar_try_wait(bar, parity);
    if (__all_sync(0xffffffffu, done)) return true;
    uint64_t el = globaltimer_ns() - t0;
    el = __shfl_sync(0xffffffffu, el, 0);
    if (el > limit_ns) return false;
  }
}

// TMA tensor store of a 3-D box (x = column, y = row, z = split) from
// shared memory, as one bulk async-group of the issuing thread.
__device__ __forceinline__ void tma_store_3d(const CUtensorMap* map, const void* src, int x, int y,
                                             int z) {
  asm volatile(
      "cp.async.bulk.tensor.3d.global.shared::cta.bulk_group [%0, {%2, %3, %4}], [%1];" ::"l"(
          reinterpret_cast<uint64_t>(map)),
      "r"(smem_u32(src)), "r"(x), "r"(y), "r"(z)
      : "memory");
}
__device__ __forceinline__ void bulk_commit() { asm volatile("cp.async.bulk.commit_group;" ::: "memory"); }
// this thread's bulk groups but the newest have finished reading shared memory
__device__ __forceinline__ void bulk_wait_read_all_but_one() {
  asm volatile("cp.async.bulk.wait_group.read 1;" ::: "memory");
}
__device__ __forceinline__ void bulk_wait_all() { asm volatile("cp.async.bulk.wait_group 0;" ::: "memory"); }
// generic-proxy writes to shared memory are visible to the async proxy (TMA)
__device__ __forceinline__ void fence_async_smem() {
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}

constexpr int kOutRows = 32;                     // rows per epilogue warp (its TMEM lanes)
constexpr int kOutChunkBytes = kOutRows * 128;   // one staged chunk: 32 rows x 128 bytes
constexpr int kOutStaging = 4 * 2 * kOutChunkBytes;  // 4 warps x 2 buffers

// Two accumulators (one per tile in flight), power-of-two column count.
template <int BN>
__host__ __device__ constexpr uint32_t tmem_cols() {
  return 2 * BN <= 32 ? 32u : (2 * BN <= 64 ? 64u : (2 * BN <= 128 ? 128u : (2 * BN <= 256 ? 256u : 512u)));
}

template <int BN, bool TMA_OUT = false>
__host__ __device__ constexpr size_t smem_bytes() {
  return 1024 /* alignment slack */ + (size_t)kStages * (BM * BK * 2 + BN * BK * 2) +
         (TMA_OUT ? kOutStaging : 0) + 256;
}

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

PFN_cuTensorMapEncodeTiled_v12000 encode_fn() {
  static std::once_flag once;
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  std::call_once(once, [] {
    cudaDriverEntryPointQueryResult q;
    void* p = nullptr;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault,
                                         &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
  });
  return fn;
}

// Tensor map of a bf16 row-major [rows, cols] matrix read as box_rows x 64
// tiles (box_cols = 64 elements = 128 bytes across a row) with 128-byte
// swizzle; out-of-range elements read as zero.  A K-major operand is read
// as rows of its M/N index; an MN-major one as 64 x 64 boxes.
bool make_map(CUtensorMap* map, const void* base, int64_t rows, int64_t cols, int box_rows) {
  auto fn = encode_fn();
  if (!fn) return false;
  const cuuint64_t dims[2] = {(cuuint64_t)cols, (cuuint64_t)rows};
  const cuuint64_t strides[1] = {(cuuint64_t)cols * 2};
  const cuuint32_t box[2] = {64u, (cuuint32_t)box_rows};
  const cuuint32_t estr[2] = {1, 1};
  return fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box,
            estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
            CU_TENSOR_MAP_L2_PROMOTION_L2_128B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// Tensor map of the output D [S, M, N] (S split partials, N contiguous;
// bf16 or fp32) written as 32-row x 128-byte boxes with 128-byte swizzle.
bool make_out_map(CUtensorMap* map, void* D, int64_t S, int64_t M, int64_t N, bool bf16) {
  auto fn = encode_fn();
  if (!fn) return false;
  const int64_t es = bf16 ? 2 : 4;
  const cuuint64_t dims[3] = {(cuuint64_t)N, (cuuint64_t)M, (cuuint64_t)S};
  const cuuint64_t strides[2] = {(cuuint64_t)(N * es), (cuuint64_t)(M * N * es)};
  const cuuint32_t box[3] = {(cuuint32_t)(128 / es), (cuuint32_t)kOutRows, 1u};
  const cuuint32_t estr[3] = {1, 1, 1};
  return fn(map, bf16 ? CU_TENSOR_MAP_DATA_TYPE_BFLOAT16 : CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 3, D,
            dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
            CU_TENSOR_MAP_L2_PROMOTION_NONE, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

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
// N tile: the widest the output needs (64 or 128 for an MN-major B), and 64
// rather than 128 when 128-wide tiles would leave most SMs idle.
template <bool OUT_BF16, bool A_MN = false, bool B_MN = false>
cudaError_t gemm_tn(const void* A, const void* B, void* D, int M, int N, int K, int* status,
                    cudaStream_t st, int ksplit = 1) {
  // a 128 x 256 tile keeps the tensor core busier per instruction (about
  // 1.6x the rate of 128 x 128 at large K); below K = 512 the per-tile
  // fixed costs dominate and the narrower tile's parallelism wins
  int bn = (!B_MN && N > 128 && K >= 512) ? 256 : 128;
  if (N <= 16 && !B_MN) bn = 16;
  else if (N <= 32 && !B_MN) bn = 32;
  else if (N <= 64) bn = 64;
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
constexpr int64_t kSplitSlots = 152;
constexpr int64_t kMinSplitKBlocks = 8;
int dw_splits(int64_t M, int64_t K, int64_t N) {
  const int64_t tiles = ((N + BM - 1) / BM) * ((K + 63) / 64);
  const int64_t nk = (M + BK - 1) / BK;
  int64_t s = kSplitSlots / (tiles > 0 ? tiles : 1);
  if (s > nk / kMinSplitKBlocks) s = nk / kMinSplitKBlocks;
  return s < 1 ? 1 : (int)s;
}

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
    const int S = dw_splits(M, K, N);
    if (M == 0) {
      e = cudaMemsetAsync(dW, 0, (size_t)N * K * sizeof(float), st);
    } else if (S == 1) {
      e = gemm_tn<false, true, true>(dI, X, dW, (int)N, (int)K, (int)M, status, st);
    } else {
      float* part = reinterpret_cast<float*>(static_cast<unsigned char*>(ws) + 256);
      e = gemm_tn<false, true, true>(dI, X, part, (int)N, (int)K, (int)M, status, st, S);
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
