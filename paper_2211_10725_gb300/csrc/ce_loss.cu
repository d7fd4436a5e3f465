// Rate-coded readout loss (Sec. V-A: the predicted class is the output
// neuron with the most spikes): cross-entropy on the spike counts over T,
// and its gradient with respect to every output spike.
//   counts[b, c] = sum_t spk[t, b, c]
//   loss = mean_b ( logsumexp_c counts[b, :] - counts[b, y_b] )
//   dL/dspk[t, b, c] = (softmax(counts[b, :])_c - [c == y_b]) / B   (same for all t)
#include <cuda_bf16.h>
#include <cuda_fp16.h>
#include <cuda_runtime.h>

#include "snn.h"
#include "snn_device.cuh"

namespace snn {
namespace {

constexpr int kCeThreads = 256;
constexpr int kMaxClasses = 1024;

// One block: thread b handles samples b, b + blockDim, ...; the loss is a
// fixed-order fp64 block sum (deterministic).
template <typename T>
__global__ void __launch_bounds__(kCeThreads) rate_ce_kernel(int64_t Tn, int64_t B, int64_t C,
                                                             int64_t ld, const T* spk,
                                                             const int* labels, float* loss,
                                                             T* grad) {
  __shared__ double sh[kCeThreads];
  double acc = 0.0;
  for (int64_t b = threadIdx.x; b < B; b += blockDim.x) {
    float cnt[32];
    float m = -1e30f;
    const int y = labels[b];
    // classes in chunks of 32 registers: pass 1 max, pass 2 sum, pass 3 grads
    for (int64_t c0 = 0; c0 < C; c0 += 32) {
      for (int j = 0; j < 32 && c0 + j < C; ++j) {
        float s = 0.0f;
        for (int64_t t = 0; t < Tn; ++t) s += Elem<T>::load1(spk + (t * B + b) * ld + c0 + j);
        m = fmaxf(m, s);
      }
    }
    double sum = 0.0;
    float cy = 0.0f;
    for (int64_t c0 = 0; c0 < C; c0 += 32) {
      for (int j = 0; j < 32 && c0 + j < C; ++j) {
        float s = 0.0f;
        for (int64_t t = 0; t < Tn; ++t) s += Elem<T>::load1(spk + (t * B + b) * ld + c0 + j);
        cnt[j] = s;
        sum += exp((double)(s - m));
        if (c0 + j == y) cy = s;
      }
    }
    const double lse = (double)m + log(sum);
    acc += lse - (double)cy;
    for (int64_t c0 = 0; c0 < C; c0 += 32) {
      for (int j = 0; j < 32 && c0 + j < C; ++j) {
        float s = 0.0f;
        for (int64_t t = 0; t < Tn; ++t) s += Elem<T>::load1(spk + (t * B + b) * ld + c0 + j);
        cnt[j] = s;
        const double p = exp((double)s - lse);
        const float gv = (float)((p - (c0 + j == y ? 1.0 : 0.0)) / (double)B);
        for (int64_t t = 0; t < Tn; ++t) Elem<T>::store1(grad + (t * B + b) * ld + c0 + j, gv);
      }
    }
    for (int64_t c = C; c < ld; ++c)
      for (int64_t t = 0; t < Tn; ++t) Elem<T>::store1(grad + (t * B + b) * ld + c, 0.0f);
  }
  sh[threadIdx.x] = acc;
  __syncthreads();
  for (int s = blockDim.x / 2; s > 0; s >>= 1) {
    if ((int)threadIdx.x < s) sh[threadIdx.x] += sh[threadIdx.x + s];
    __syncthreads();
  }
  if (threadIdx.x == 0) loss[0] = (float)(sh[0] / (double)(B > 0 ? B : 1));
}

}  // namespace
}  // namespace snn

extern "C" snn_status_t snn_rate_ce_loss(int64_t T, int64_t B, int64_t C, int64_t ld, int32_t dtype,
                                         const void* spk, const int32_t* labels, float* loss,
                                         void* grad_spk, snn_stream_t stream) {
  if (T < 0 || B < 0 || C < 1 || ld < C || C > snn::kMaxClasses) return SNN_ERR_INVALID_ARG;
  if (!loss || (T > 0 && B > 0 && (!spk || !labels || !grad_spk))) return SNN_ERR_INVALID_ARG;
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  switch (dtype) {
    case SNN_F32:
      snn::rate_ce_kernel<float><<<1, snn::kCeThreads, 0, st>>>(
          T, B, C, ld, static_cast<const float*>(spk), labels, loss, static_cast<float*>(grad_spk));
      break;
    case SNN_BF16:
      snn::rate_ce_kernel<__nv_bfloat16><<<1, snn::kCeThreads, 0, st>>>(
          T, B, C, ld, static_cast<const __nv_bfloat16*>(spk), labels, loss,
          static_cast<__nv_bfloat16*>(grad_spk));
      break;
    case SNN_F16:
      snn::rate_ce_kernel<__half><<<1, snn::kCeThreads, 0, st>>>(
          T, B, C, ld, static_cast<const __half*>(spk), labels, loss, static_cast<__half*>(grad_spk));
      break;
    default:
      return SNN_ERR_INVALID_ARG;
  }
  return cudaGetLastError() == cudaSuccess ? SNN_OK : SNN_ERR_CUDA;
}
