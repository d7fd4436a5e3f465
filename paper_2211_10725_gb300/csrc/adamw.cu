// AdamW update of the dense weights (the optimiser of the paper's training
// runs, Sec. V): decoupled weight decay plus the bias-corrected Adam step,
//   m <- b1 m + (1 - b1) g,   v <- b2 v + (1 - b2) g^2
//   w <- w (1 - lr wd) - (lr / c1) m / (sqrt(v / c2) + eps),  c_i = 1 - b_i^step
// on fp32 master weights, with an optional bf16 copy of the result written
// for the next forward GEMM.  Elementwise: each thread moves four elements
// with 16-byte accesses; a scalar loop covers the tail.
//
// The step number comes from the host, or from a device counter that the
// launch itself advances, so that a captured CUDA graph replays successive
// steps: every block reads the counter first, and the last block to finish
// (a ticket taken after the read) writes the next value.
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include <algorithm>
#include <cmath>
#include <cstdint>

#include "launch.cuh"
#include "snn.h"

namespace snn {
namespace {

constexpr int kAdamThreads = 256;

struct AdamCoef {
  float b1, b2, one_m_b1, one_m_b2, decay, step_size, rsqrt_c2, eps;
};

struct AdamHyper {
  double lr, b1, b2;
};

// Bias-corrected step size and 1/sqrt(1 - beta2^step): 1 - beta^step as
// -expm1(step * log(beta)), which keeps its precision at small step.  The
// host evaluates it in double; the device (counter mode, once per block) in
// float, since double arithmetic is slow on this part.
inline void bias_terms_host(const AdamHyper& h, int64_t step, AdamCoef& c) {
  const double c1 = -std::expm1((double)step * std::log(h.b1));
  const double c2 = -std::expm1((double)step * std::log(h.b2));
  c.step_size = (float)(h.lr / c1);
  c.rsqrt_c2 = (float)(1.0 / std::sqrt(c2));
}

__device__ __forceinline__ void bias_terms_device(const AdamHyper& h, uint64_t step, AdamCoef& c) {
  const float s = (float)step;
  const float c1 = -expm1f(s * logf((float)h.b1));
  const float c2 = -expm1f(s * logf((float)h.b2));
  c.step_size = (float)h.lr / c1;
  c.rsqrt_c2 = 1.0f / sqrtf(c2);
}

__device__ __forceinline__ float adam_one(float w, float g, float& m, float& v, const AdamCoef& c) {
  m = __fmaf_rn(c.b1, m, c.one_m_b1 * g);
  v = __fmaf_rn(c.b2, v, c.one_m_b2 * (g * g));
  const float denom = sqrtf(v) * c.rsqrt_c2 + c.eps;
  return w * c.decay - c.step_size * (m / denom);
}

__global__ void __launch_bounds__(kAdamThreads) adamw_kernel(int64_t n, float* __restrict__ w,
                                                             __nv_bfloat16* __restrict__ wl,
                                                             const float* __restrict__ g,
                                                             float* __restrict__ m,
                                                             float* __restrict__ v, AdamCoef c,
                                                             AdamHyper h,
                                                             unsigned long long* counter) {
  grid_dep_wait();
  if (counter) {
    // counter[0]: updates done so far; counter[1]: blocks finished reading
    __shared__ AdamCoef sc;
    if (threadIdx.x == 0) {
      const unsigned long long done = *reinterpret_cast<volatile unsigned long long*>(counter);
      sc = c;
      bias_terms_device(h, done + 1, sc);
      __threadfence();
      const unsigned long long ticket = atomicAdd(counter + 1, 1ull);
      if (ticket == gridDim.x - 1) {  // every block has read counter[0]
        counter[0] = done + 1;
        counter[1] = 0;
      }
    }
    __syncthreads();
    c = sc;
  }
  const int64_t n4 = n / 4;
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n4; i += stride) {
    float4 wv = reinterpret_cast<float4*>(w)[i];
    const float4 gv = reinterpret_cast<const float4*>(g)[i];
    float4 mv = reinterpret_cast<float4*>(m)[i];
    float4 vv = reinterpret_cast<float4*>(v)[i];
    wv.x = adam_one(wv.x, gv.x, mv.x, vv.x, c);
    wv.y = adam_one(wv.y, gv.y, mv.y, vv.y, c);
    wv.z = adam_one(wv.z, gv.z, mv.z, vv.z, c);
    wv.w = adam_one(wv.w, gv.w, mv.w, vv.w, c);
    reinterpret_cast<float4*>(w)[i] = wv;
    reinterpret_cast<float4*>(m)[i] = mv;
    reinterpret_cast<float4*>(v)[i] = vv;
    if (wl) {
      __nv_bfloat162 lo = __floats2bfloat162_rn(wv.x, wv.y);
      __nv_bfloat162 hi = __floats2bfloat162_rn(wv.z, wv.w);
      uint2 pack;
      pack.x = *reinterpret_cast<unsigned*>(&lo);
      pack.y = *reinterpret_cast<unsigned*>(&hi);
      reinterpret_cast<uint2*>(wl)[i] = pack;
    }
  }
  for (int64_t i = 4 * n4 + (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += stride) {
    float mi = m[i], vi = v[i];
    const float wi = adam_one(w[i], g[i], mi, vi, c);
    w[i] = wi;
    m[i] = mi;
    v[i] = vi;
    if (wl) wl[i] = __float2bfloat16_rn(wi);
  }
}

}  // namespace
}  // namespace snn

extern "C" snn_status_t snn_adamw_step(int64_t n, float* w, void* w_bf16, const float* grad,
                                       float* m, float* v, float lr, float beta1, float beta2,
                                       float eps, float weight_decay, int64_t step,
                                       int64_t* step_counter, snn_stream_t stream) {
  if (n < 0 || (!step_counter && step < 1)) return SNN_ERR_INVALID_ARG;
  if (step_counter && (reinterpret_cast<uintptr_t>(step_counter) & 15u)) return SNN_ERR_ALIGNMENT;
  if (!(beta1 > 0.0f && beta1 < 1.0f && beta2 > 0.0f && beta2 < 1.0f && eps > 0.0f))
    return SNN_ERR_INVALID_ARG;
  if (n == 0) return SNN_OK;
  if (!w || !grad || !m || !v) return SNN_ERR_INVALID_ARG;
  const void* ptrs[5] = {w, grad, m, v, w_bf16};
  for (const void* p : ptrs)
    if (reinterpret_cast<uintptr_t>(p) & 15u) return SNN_ERR_ALIGNMENT;
  snn::AdamCoef c;
  c.b1 = beta1;
  c.b2 = beta2;
  c.one_m_b1 = 1.0f - beta1;
  c.one_m_b2 = 1.0f - beta2;
  c.decay = (float)(1.0 - (double)lr * (double)weight_decay);
  c.eps = eps;
  const snn::AdamHyper h{(double)lr, (double)beta1, (double)beta2};
  snn::bias_terms_host(h, step_counter ? 1 : step, c);
  int dev = 0, sms = 152;
  if (cudaGetDevice(&dev) == cudaSuccess)
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  const int64_t want = (n / 4 + snn::kAdamThreads - 1) / snn::kAdamThreads;
  const int blocks = (int)std::max<int64_t>(1, std::min<int64_t>(want, (int64_t)sms * 8));
  const cudaError_t e = snn::launch_pdl(
      snn::adamw_kernel, dim3(blocks), dim3(snn::kAdamThreads), 0,
      reinterpret_cast<cudaStream_t>(stream), n, w, static_cast<__nv_bfloat16*>(w_bf16), grad, m,
      v, c, h, reinterpret_cast<unsigned long long*>(step_counter));
  return e == cudaSuccess ? SNN_OK : SNN_ERR_CUDA;
}
