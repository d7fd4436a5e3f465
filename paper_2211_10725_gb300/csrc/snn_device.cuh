// Device-side building blocks of libsnn: inline-PTX wrappers for mbarriers
// and bulk (TMA) copies, bounded waits, element conversion.
#pragma once

#include <cuda_bf16.h>
#include <cuda_fp16.h>
#include <cuda_runtime.h>
#include <stdint.h>

namespace snn {

// Status values written into the workspace word (match snn_status_t).
constexpr int kStatusTimeout = 6;

// ---------------------------------------------------------------------------
// Shared-memory addresses, mbarriers, bulk copies
// ---------------------------------------------------------------------------

__device__ __forceinline__ uint32_t smem_u32(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ void mbar_init(uint64_t* bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_u32(bar)), "r"(count)
               : "memory");
}

// Make barrier initialisation visible to the async (TMA) proxy.
__device__ __forceinline__ void fence_barrier_init() {
  asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}

__device__ __forceinline__ void mbar_arrive(uint64_t* bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(smem_u32(bar)) : "memory");
}

__device__ __forceinline__ void mbar_arrive_expect_tx(uint64_t* bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_u32(bar)),
               "r"(bytes)
               : "memory");
}

__device__ __forceinline__ bool mbar_try_wait(uint64_t* bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(ok)
      : "r"(smem_u32(bar)), "r"(parity)
      : "memory");
  return ok != 0;
}

// As mbar_try_wait, but the thread may stay suspended in the instruction for
// up to hint_ns (it resumes when the phase completes): for waits off the
// critical path, so that polling does not take issue slots from other warps.
__device__ __forceinline__ bool mbar_try_wait_sleep(uint64_t* bar, uint32_t parity,
                                                    uint32_t hint_ns) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2, %3;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(ok)
      : "r"(smem_u32(bar)), "r"(parity), "r"(hint_ns)
      : "memory");
  return ok != 0;
}

__device__ __forceinline__ uint64_t globaltimer_ns() {
  uint64_t t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}

// Wait for the phase of `bar` with the given parity to complete, for at most
// limit_ns nanoseconds.  Returns false if the wait gave up.
__device__ __forceinline__ bool mbar_wait_bounded(uint64_t* bar, uint32_t parity,
                                                  uint64_t limit_ns) {
  if (mbar_try_wait(bar, parity)) return true;
  const uint64_t t0 = globaltimer_ns();
  while (!mbar_try_wait_sleep(bar, parity, 20000u)) {
    if (globaltimer_ns() - t0 > limit_ns) return false;
  }
  return true;
}

// Bounded wait of a single thread on a critical path (a producer refilling
// a ring stage): polls without the suspend hint -- a thread suspended in
// try_wait can resume microseconds after the phase completes, which starves
// a shallow ring -- and reads the clock only every 64 polls.
__device__ __forceinline__ bool mbar_wait_spin(uint64_t* bar, uint32_t parity, uint64_t limit_ns) {
  if (mbar_try_wait(bar, parity)) return true;
  const uint64_t t0 = globaltimer_ns();
  for (uint32_t i = 1;; ++i) {
    if (mbar_try_wait(bar, parity)) return true;
    if ((i & 63u) == 0 && globaltimer_ns() - t0 > limit_ns) return false;
  }
}

// 1-D bulk copy global -> this CTA's shared memory, completing `bytes` of
// transaction count on `bar`.  dst, src and bytes are multiples of 16.
__device__ __forceinline__ void bulk_g2s(void* dst, const void* src, uint32_t bytes,
                                         uint64_t* bar) {
  asm volatile(
      "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
          smem_u32(dst)),
      "l"(src), "r"(bytes), "r"(smem_u32(bar))
      : "memory");
}

__device__ __forceinline__ void record_status(int* status, int code) {
  if (status) atomicCAS(status, 0, code);
}

// ---------------------------------------------------------------------------
// Element conversion: 8 or 4 consecutive elements <-> float[], or one element
// ---------------------------------------------------------------------------

template <typename T>
struct Elem;

template <>
struct Elem<float> {
  static __device__ __forceinline__ void load8(const float* p, float v[8]) {
    const float4 a = reinterpret_cast<const float4*>(p)[0];
    const float4 b = reinterpret_cast<const float4*>(p)[1];
    v[0] = a.x; v[1] = a.y; v[2] = a.z; v[3] = a.w;
    v[4] = b.x; v[5] = b.y; v[6] = b.z; v[7] = b.w;
  }
  static __device__ __forceinline__ void store8(float* p, const float v[8]) {
    reinterpret_cast<float4*>(p)[0] = make_float4(v[0], v[1], v[2], v[3]);
    reinterpret_cast<float4*>(p)[1] = make_float4(v[4], v[5], v[6], v[7]);
  }
  static __device__ __forceinline__ void load4(const float* p, float v[4]) {
    const float4 a = *reinterpret_cast<const float4*>(p);
    v[0] = a.x; v[1] = a.y; v[2] = a.z; v[3] = a.w;
  }
  static __device__ __forceinline__ void store4(float* p, const float v[4]) {
    *reinterpret_cast<float4*>(p) = make_float4(v[0], v[1], v[2], v[3]);
  }
  static __device__ __forceinline__ float load1(const float* p) { return *p; }
  static __device__ __forceinline__ void store1(float* p, float v) { *p = v; }
};

template <>
struct Elem<__nv_bfloat16> {
  static __device__ __forceinline__ float2 to2(uint32_t w) {
    return __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(&w));
  }
  static __device__ __forceinline__ uint32_t from2(float a, float b) {
    __nv_bfloat162 h = __floats2bfloat162_rn(a, b);
    return *reinterpret_cast<uint32_t*>(&h);
  }
  static __device__ __forceinline__ void load8(const __nv_bfloat16* p, float v[8]) {
    const uint4 x = *reinterpret_cast<const uint4*>(p);
    float2 f;
    f = to2(x.x); v[0] = f.x; v[1] = f.y;
    f = to2(x.y); v[2] = f.x; v[3] = f.y;
    f = to2(x.z); v[4] = f.x; v[5] = f.y;
    f = to2(x.w); v[6] = f.x; v[7] = f.y;
  }
  static __device__ __forceinline__ void store8(__nv_bfloat16* p, const float v[8]) {
    *reinterpret_cast<uint4*>(p) =
        make_uint4(from2(v[0], v[1]), from2(v[2], v[3]), from2(v[4], v[5]), from2(v[6], v[7]));
  }
  static __device__ __forceinline__ void load4(const __nv_bfloat16* p, float v[4]) {
    const uint2 x = *reinterpret_cast<const uint2*>(p);
    float2 f;
    f = to2(x.x); v[0] = f.x; v[1] = f.y;
    f = to2(x.y); v[2] = f.x; v[3] = f.y;
  }
  static __device__ __forceinline__ void store4(__nv_bfloat16* p, const float v[4]) {
    *reinterpret_cast<uint2*>(p) = make_uint2(from2(v[0], v[1]), from2(v[2], v[3]));
  }
  static __device__ __forceinline__ float load1(const __nv_bfloat16* p) {
    return __bfloat162float(*p);
  }
  static __device__ __forceinline__ void store1(__nv_bfloat16* p, float v) {
    *p = __float2bfloat16_rn(v);
  }
};

template <>
struct Elem<__half> {
  static __device__ __forceinline__ float2 to2(uint32_t w) {
    return __half22float2(*reinterpret_cast<const __half2*>(&w));
  }
  static __device__ __forceinline__ uint32_t from2(float a, float b) {
    __half2 h = __floats2half2_rn(a, b);
    return *reinterpret_cast<uint32_t*>(&h);
  }
  static __device__ __forceinline__ void load8(const __half* p, float v[8]) {
    const uint4 x = *reinterpret_cast<const uint4*>(p);
    float2 f;
    f = to2(x.x); v[0] = f.x; v[1] = f.y;
    f = to2(x.y); v[2] = f.x; v[3] = f.y;
    f = to2(x.z); v[4] = f.x; v[5] = f.y;
    f = to2(x.w); v[6] = f.x; v[7] = f.y;
  }
  static __device__ __forceinline__ void store8(__half* p, const float v[8]) {
    *reinterpret_cast<uint4*>(p) =
        make_uint4(from2(v[0], v[1]), from2(v[2], v[3]), from2(v[4], v[5]), from2(v[6], v[7]));
  }
  static __device__ __forceinline__ void load4(const __half* p, float v[4]) {
    const uint2 x = *reinterpret_cast<const uint2*>(p);
    float2 f;
    f = to2(x.x); v[0] = f.x; v[1] = f.y;
    f = to2(x.y); v[2] = f.x; v[3] = f.y;
  }
  static __device__ __forceinline__ void store4(__half* p, const float v[4]) {
    *reinterpret_cast<uint2*>(p) = make_uint2(from2(v[0], v[1]), from2(v[2], v[3]));
  }
  static __device__ __forceinline__ float load1(const __half* p) { return __half2float(*p); }
  static __device__ __forceinline__ void store1(__half* p, float v) { *p = __float2half_rn(v); }
};

// V consecutive elements (V = 4 or 8), aligned to V elements
template <typename T, int V>
__device__ __forceinline__ void loadv(const T* p, float* v) {
  static_assert(V == 4 || V == 8, "vector accesses of 4 or 8 elements");
  if constexpr (V == 8) Elem<T>::load8(p, v);
  else Elem<T>::load4(p, v);
}
template <typename T, int V>
__device__ __forceinline__ void storev(T* p, const float* v) {
  static_assert(V == 4 || V == 8, "vector accesses of 4 or 8 elements");
  if constexpr (V == 8) Elem<T>::store8(p, v);
  else Elem<T>::store4(p, v);
}

}  // namespace snn
