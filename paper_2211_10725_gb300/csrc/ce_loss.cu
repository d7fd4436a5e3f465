// Rate-coded readout loss (Sec. V-A: the predicted class is the output
// neuron with the most spikes): cross-entropy on the spike counts over T,
// and its gradient with respect to every output spike.
//   counts[b, c] = sum_t sum_j spk[t, b, c*pop + j]   (j < pop: the class's
//                  population, Sec. VII; pop = 1 is the plain rate code)
//   loss = sum_b ( logsumexp_c counts[b, :] - counts[b, y_b] ) / B_norm
//   dL/dspk[t, b, c*pop + j] = (softmax(counts[b, :])_c - [c == y_b]) / B_norm
//                  (the same for every t and every neuron of the population)
// B_norm is the batch the mean is taken over: B, or the global batch when
// B samples are one data-parallel shard (the shards' results then add up to
// the global loss and gradient).
//
// One block per sample:
//   1. the threads sum spk over t for the sample's neurons (t in order,
//      eight time steps' loads in flight per thread) into shared counts;
//   2. the threads add each class's population counts in order;
//   3. warp 0 takes the softmax over the classes (lanes over c) and writes
//      the sample's loss term to the workspace; the class gradients replace
//      the class counts;
//   4. the threads write the gradient of every neuron for every t.
// The last block to finish (a ticket taken after its loss term is
// published) adds the B loss terms in sample order: deterministic.  The
// softmax runs in float (double arithmetic is slow on this part); the loss
// terms and their sum are in double.
#include <cuda_bf16.h>
#include <cuda_fp16.h>
#include <cuda_runtime.h>

#include <climits>

#include "scan_host.cuh"
#include "snn.h"

namespace snn {
namespace {

constexpr int kCeThreads = 256;
constexpr int kMaxClasses = 1024;
constexpr int kCeMaxNeurons = 32 * 1024;  // C*pop: counts held in shared memory

__device__ __forceinline__ float warp_max(float v) {
  for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
  return v;
}

__device__ __forceinline__ float warp_sum(float v) {
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

template <typename T>
__global__ void __launch_bounds__(kCeThreads) rate_ce_kernel(int64_t Tn, int64_t B, int C,
                                                             int pop, int64_t ld, int64_t Bn,
                                                             const T* spk, const int* labels,
                                                             float* loss, T* grad, double* terms,
                                                             int* ticket) {
  extern __shared__ __align__(16) float ce_smem[];
  const int CP = C * pop;
  float* ncnt = ce_smem;       // [CP] neuron counts
  float* ccnt = ce_smem + CP;  // [C] class counts, then class gradients
  __shared__ int last;
  grid_dep_wait();
  const int64_t b = blockIdx.x;
  const int64_t step = B * ld;
  const T* row = spk + b * ld;
  for (int n = threadIdx.x; n < CP; n += kCeThreads) {
    const T* p = row + n;
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
    ncnt[n] = s;
  }
  __syncthreads();
  for (int c = threadIdx.x; c < C; c += kCeThreads) {
    float s = 0.0f;
    for (int k = 0; k < pop; ++k) s += ncnt[c * pop + k];
    ccnt[c] = s;
  }
  __syncthreads();
  if (threadIdx.x < 32) {
    const int lane = threadIdx.x;
    const int y = labels[b];
    float m = -1e30f;
    for (int c = lane; c < C; c += 32) m = fmaxf(m, ccnt[c]);
    m = warp_max(m);
    float se = 0.0f, cy = 0.0f;
    for (int c = lane; c < C; c += 32) {
      se += expf(ccnt[c] - m);
      if (c == y) cy = ccnt[c];
    }
    se = warp_sum(se);
    cy = warp_sum(cy);
    // loss = (m - count_y) + log(sum_c exp(count_c - m)); softmax_c =
    // exp(count_c - m) / sum, both relative to the largest count
    if (lane == 0) terms[b] = (double)(m - cy) + (double)logf(se);
    __syncwarp();
    const float inv_b = 1.0f / (float)Bn;
    for (int c = lane; c < C; c += 32)
      ccnt[c] = (expf(ccnt[c] - m) / se - (c == y ? 1.0f : 0.0f)) * inv_b;
  }
  __syncthreads();
  T* grow = grad + b * ld;
  for (int64_t n = threadIdx.x; n < ld; n += kCeThreads) {
    const float g = n < CP ? ccnt[n / pop] : 0.0f;
    for (int64_t t = 0; t < Tn; ++t) Elem<T>::store1(grow + t * step + n, g);
  }
  // the last block to finish adds the loss terms in sample order
  __threadfence();
  __syncthreads();
  if (threadIdx.x == 0) last = atomicAdd(ticket, 1) == (int)(B - 1);
  __syncthreads();
  if (!last) return;
  __threadfence();
  if (threadIdx.x == 0) {
    double total = 0.0;
    for (int64_t q = 0; q < B; ++q) total += terms[q];
    loss[0] = (float)(total / (double)Bn);
    *ticket = 0;
  }
}

template <typename T>
cudaError_t launch_ce(int64_t Tn, int64_t B, int C, int pop, int64_t ld, int64_t Bn,
                      const void* spk, const int* labels, float* loss, void* grad, double* terms,
                      int* ticket, cudaStream_t st) {
  const size_t smem = (size_t)(C * pop + C) * sizeof(float);
  const void* k = (const void*)rate_ce_kernel<T>;
  const cudaError_t e = ensure_smem(k, smem);
  if (e != cudaSuccess) return e;
  return launch_pdl(rate_ce_kernel<T>, dim3((unsigned)B), dim3(kCeThreads), smem, st, Tn, B, C,
                    pop, ld, Bn, static_cast<const T*>(spk), labels, loss, static_cast<T*>(grad),
                    terms, ticket);
}

}  // namespace
}  // namespace snn

extern "C" size_t snn_rate_ce_workspace_bytes(int64_t B) {
  if (B < 0 || B > INT_MAX) return 0;
  return 256 + (size_t)B * sizeof(double);
}

extern "C" snn_status_t snn_rate_ce_loss(int64_t T, int64_t B, int64_t C, int64_t pop, int64_t ld,
                                         int64_t batch_total, int32_t dtype, const void* spk,
                                         const int32_t* labels, float* loss, void* grad_spk,
                                         void* ws, size_t ws_bytes, snn_stream_t stream) {
  if (T < 0 || B < 0 || B > INT_MAX || C < 1 || pop < 1 || C > snn::kMaxClasses)
    return SNN_ERR_INVALID_ARG;
  if (pop > snn::kCeMaxNeurons / C || ld < C * pop) return SNN_ERR_INVALID_ARG;
  const int64_t Bn = batch_total > 0 ? batch_total : (B > 0 ? B : 1);
  if (batch_total > 0 && batch_total < B) return SNN_ERR_INVALID_ARG;
  if (dtype != SNN_F32 && dtype != SNN_BF16 && dtype != SNN_F16) return SNN_ERR_INVALID_ARG;
  if (!loss || (T > 0 && B > 0 && (!spk || !labels || !grad_spk))) return SNN_ERR_INVALID_ARG;
  if (!ws || ws_bytes < snn_rate_ce_workspace_bytes(B)) return SNN_ERR_WORKSPACE;
  if (reinterpret_cast<uintptr_t>(ws) & 15u) return SNN_ERR_ALIGNMENT;
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  if (B == 0)
    return cudaMemsetAsync(loss, 0, sizeof(float), st) == cudaSuccess ? SNN_OK : SNN_ERR_CUDA;
  unsigned char* w = static_cast<unsigned char*>(ws);
  int* ticket = reinterpret_cast<int*>(w);
  double* terms = reinterpret_cast<double*>(w + 256);
  cudaError_t e;
  switch (dtype) {
    case SNN_F32:
      e = snn::launch_ce<float>(T, B, (int)C, (int)pop, ld, Bn, spk, labels, loss, grad_spk, terms,
                                ticket, st);
      break;
    case SNN_BF16:
      e = snn::launch_ce<__nv_bfloat16>(T, B, (int)C, (int)pop, ld, Bn, spk, labels, loss,
                                        grad_spk, terms, ticket, st);
      break;
    default:
      e = snn::launch_ce<__half>(T, B, (int)C, (int)pop, ld, Bn, spk, labels, loss, grad_spk,
                                 terms, ticket, st);
  }
  return e == cudaSuccess ? SNN_OK : SNN_ERR_CUDA;
}
