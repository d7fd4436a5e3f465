// Rate-coded readout loss (Sec. V-A: the predicted class is the output
// neuron with the most spikes): cross-entropy on the spike counts over T,
// and its gradient with respect to every output spike.
//   counts[b, c] = sum_t spk[t, b, c]
//   loss = sum_b ( logsumexp_c counts[b, :] - counts[b, y_b] ) / B_norm
//   dL/dspk[t, b, c] = (softmax(counts[b, :])_c - [c == y_b]) / B_norm   (same for all t)
// B_norm is the batch the mean is taken over: B, or the global batch when
// B samples are one data-parallel shard (the shards' results then add up to
// the global loss and gradient).
#include <cuda_bf16.h>
#include <cuda_fp16.h>
#include <cuda_runtime.h>

#include "snn.h"
#include "snn_device.cuh"

namespace snn {
namespace {

constexpr int kCeThreads = 1024;
constexpr int kCeWarps = kCeThreads / 32;
constexpr int kMaxClasses = 1024;
constexpr int kCountSlots = 8192;  // shared-memory counts per chunk of samples

__device__ __forceinline__ float warp_max(float v) {
  for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
  return v;
}

__device__ __forceinline__ float warp_sum(float v) {
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

// One block, samples in chunks of Bc = kCountSlots / C:
//   1. every thread sums spk over t for (b, c) pairs of the chunk, t in a
//      fixed order (8 independent loads in flight), into shared counts;
//   2. warp w takes the chunk's samples w, w + 32, ...: softmax over the
//      classes with lanes over c, the sample's loss added to the warp's sum
//      in sample order, the gradient row written back over the counts;
//   3. every thread writes gradients of (b, c) pairs for every t, so that
//      the threads of a warp store a contiguous run of each row.
// The softmax runs in float (double arithmetic is slow on this part); each
// warp adds its samples' losses in double, and the 32 warp sums are added in
// warp order: the loss is deterministic.
template <typename T>
__global__ void __launch_bounds__(kCeThreads) rate_ce_kernel(int64_t Tn, int64_t B, int64_t C,
                                                             int64_t ld, int64_t Bn, const T* spk,
                                                             const int* labels, float* loss,
                                                             T* grad) {
  __shared__ float cnt[kCountSlots];
  __shared__ double warp_loss[kCeWarps];
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int64_t Bc = kCountSlots / C;
  const float inv_b = 1.0f / (float)Bn;
  double acc = 0.0;
  for (int64_t b0 = 0; b0 < B; b0 += Bc) {
    const int64_t nb = min(Bc, B - b0);
    for (int64_t e = threadIdx.x; e < nb * C; e += kCeThreads) {
      const int64_t b = b0 + e / C, c = e % C;
      const T* p = spk + b * ld + c;
      const int64_t step = B * ld;
      float s = 0.0f;
      int64_t t = 0;
      for (; t + 8 <= Tn; t += 8) {
        float v[8];
#pragma unroll
        for (int k = 0; k < 8; ++k) v[k] = Elem<T>::load1(p + (t + k) * step);
#pragma unroll
        for (int k = 0; k < 8; ++k) s += v[k];
      }
      for (; t < Tn; ++t) s += Elem<T>::load1(p + t * step);
      cnt[e] = s;
    }
    __syncthreads();
    for (int64_t j = warp; j < nb; j += kCeWarps) {
      float* row = cnt + j * C;
      const int y = labels[b0 + j];
      float m = -1e30f;
      for (int64_t c = lane; c < C; c += 32) m = fmaxf(m, row[c]);
      m = warp_max(m);
      float se = 0.0f, cy = 0.0f;
      for (int64_t c = lane; c < C; c += 32) {
        se += expf(row[c] - m);
        if (c == y) cy = row[c];
      }
      se = warp_sum(se);
      cy = warp_sum(cy);
      // loss = (m - count_y) + log(sum_c exp(count_c - m)); softmax_c =
      // exp(count_c - m) / sum, both relative to the largest count
      acc += (double)(m - cy) + (double)logf(se);
      __syncwarp();
      for (int64_t c = lane; c < C; c += 32)
        row[c] = (expf(row[c] - m) / se - (c == y ? 1.0f : 0.0f)) * inv_b;
    }
    __syncthreads();
    for (int64_t r = threadIdx.x; r < nb * ld; r += kCeThreads) {
      const int64_t j = r / ld, c = r - j * ld;
      const float g = c < C ? cnt[j * C + c] : 0.0f;
      T* q = grad + b0 * ld + r;
      for (int64_t t = 0; t < Tn; ++t) Elem<T>::store1(q + t * B * ld, g);
    }
    __syncthreads();
  }
  if (lane == 0) warp_loss[warp] = acc;
  __syncthreads();
  if (threadIdx.x == 0) {
    double total = 0.0;
    for (int w = 0; w < kCeWarps; ++w) total += warp_loss[w];
    loss[0] = (float)(total / (double)Bn);
  }
}

}  // namespace
}  // namespace snn

extern "C" snn_status_t snn_rate_ce_loss(int64_t T, int64_t B, int64_t C, int64_t ld,
                                         int64_t batch_total, int32_t dtype, const void* spk,
                                         const int32_t* labels, float* loss, void* grad_spk,
                                         snn_stream_t stream) {
  if (T < 0 || B < 0 || C < 1 || ld < C || C > snn::kMaxClasses) return SNN_ERR_INVALID_ARG;
  const int64_t Bn = batch_total > 0 ? batch_total : (B > 0 ? B : 1);
  if (batch_total > 0 && batch_total < B) return SNN_ERR_INVALID_ARG;
  if (!loss || (T > 0 && B > 0 && (!spk || !labels || !grad_spk))) return SNN_ERR_INVALID_ARG;
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  switch (dtype) {
    case SNN_F32:
      snn::rate_ce_kernel<float><<<1, snn::kCeThreads, 0, st>>>(
          T, B, C, ld, Bn, static_cast<const float*>(spk), labels, loss, static_cast<float*>(grad_spk));
      break;
    case SNN_BF16:
      snn::rate_ce_kernel<__nv_bfloat16><<<1, snn::kCeThreads, 0, st>>>(
          T, B, C, ld, Bn, static_cast<const __nv_bfloat16*>(spk), labels, loss,
          static_cast<__nv_bfloat16*>(grad_spk));
      break;
    case SNN_F16:
      snn::rate_ce_kernel<__half><<<1, snn::kCeThreads, 0, st>>>(
          T, B, C, ld, Bn, static_cast<const __half*>(spk), labels, loss, static_cast<__half*>(grad_spk));
      break;
    default:
      return SNN_ERR_INVALID_ARG;
  }
  return cudaGetLastError() == cudaSuccess ? SNN_OK : SNN_ERR_CUDA;
}
