// tcgen05 building blocks shared by the tensor-core kernels (the dense
// GEMM and the GEMM with a Leaky-scan epilogue): TMA tile loads and stores,
// shared-memory matrix and instruction descriptors, tcgen05.mma / commit,
// TMEM allocation and loads, bounded mbarrier waits, and the host side
// tensor-map encoders.
#pragma once

#include <cuda.h>
#include <cudaTypedefs.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include <cstdint>
#include <mutex>

#include "scan_host.cuh"

namespace snn {
namespace gemm {

#ifndef SNN_GEMM_CTAS_PER_SM
#define SNN_GEMM_CTAS_PER_SM 1
#endif
#ifndef SNN_GEMM_SLEEP_WAIT
#define SNN_GEMM_SLEEP_WAIT 0
#endif

constexpr int BM = 128;
constexpr int BK = 64;  // 64 bf16 = 128 bytes: one swizzle atom row
// Ring depth of the plain GEMM: one CTA per SM streams its operands through
// a TMA ring, and its feed rate is the bytes it has in flight, so each tile
// width takes as many stages as fit beside the output staging in the 227 KB
// a CTA may use (all three come to 225 KB with the staging).
template <int BN>
__host__ __device__ constexpr int gemm_stages() { return BN <= 64 ? 8 : (BN <= 128 ? 6 : 4); }
constexpr int kCtasPerSm = SNN_GEMM_CTAS_PER_SM;  // resident CTAs the tile size aims for
constexpr int kThreads = 192;
constexpr uint64_t kDefaultWaitNs = 2000000000ull;
constexpr uint64_t kDrainWaitNs = 1000000000ull;


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

// 3-D tile load (x innermost), e.g. rows of several time steps at once.
__device__ __forceinline__ void tma_load_3d(void* dst, const CUtensorMap* map, int x, int y, int z,
                                            uint64_t* bar) {
  asm volatile(
      "cp.async.bulk.tensor.3d.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3, %4}], [%5];" ::"r"(
          smem_u32(dst)),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(z), "r"(smem_u32(bar))
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
  return mbar_wait_spin(bar, parity, limit_ns);
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
  return 1024 /* alignment slack */ + (size_t)gemm_stages<BN>() * (BM * BK * 2 + BN * BK * 2) +
         (TMA_OUT ? kOutStaging : 0) + 256;
}

// ---------------------------------------------------------------------------
// Host side: tensor maps
// ---------------------------------------------------------------------------

inline PFN_cuTensorMapEncodeTiled_v12000 encode_fn() {
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
inline bool make_map(CUtensorMap* map, const void* base, int64_t rows, int64_t cols, int box_rows) {
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
inline bool make_out_map(CUtensorMap* map, void* D, int64_t S, int64_t M, int64_t N, bool bf16) {
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

// Tensor map of a bf16 [T, R, K] tensor (K contiguous) read as boxes of 64
// (K) x rows (R) x steps (T) with 128-byte swizzle: the box lands in shared
// memory as rows*steps 128-byte rows ordered (t, r).
inline bool make_map_3d(CUtensorMap* map, const void* base, int64_t T, int64_t R, int64_t K,
                        int box_rows, int box_steps) {
  auto fn = encode_fn();
  if (!fn) return false;
  const cuuint64_t dims[3] = {(cuuint64_t)K, (cuuint64_t)R, (cuuint64_t)T};
  const cuuint64_t strides[2] = {(cuuint64_t)K * 2, (cuuint64_t)(R * K * 2)};
  const cuuint32_t box[3] = {64u, (cuuint32_t)box_rows, (cuuint32_t)box_steps};
  const cuuint32_t estr[3] = {1, 1, 1};
  return fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(base), dims, strides, box,
            estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
            CU_TENSOR_MAP_L2_PROMOTION_L2_128B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

}  // namespace gemm
}  // namespace snn
