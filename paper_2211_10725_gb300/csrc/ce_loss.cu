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
// published) adds the B loss terms in a fixed order (strided per thread,
// then by warps): deterministic.  The
// softmax runs in float (double arithmetic is slow on this part); the loss
// terms and their sum are in double.
//
// With the readout's BPTT (snn_rate_ce_leaky_bwd), step 4 also runs the
// output layer's reverse scan (Sec. III-B) for each of the sample's neurons
// on its stored trace: the spike gradient is the constant of step 3, so
// dL/dI of the readout comes out of the same launch.
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

// The readout layer's stored state and parameters for the fused BPTT.
template <typename T>
struct ReadoutBptt {
  ScanArgs sa;            // reset, detach and surrogate of bwd_step
  const float* beta;      // scalar (beta_col 0) or one per neuron of ld
  const float* thr;
  int beta_col, thr_col;
  const T* mem;           // [T, B, ld] stored trace
  const unsigned char* bits;  // spike bits (store-mode layout), or null: z from spk
  int64_t bits_row;
  T* gI;                  // [T, B, ld] dL/dI
};

constexpr int kCeChunk = 8;  // steps of stored trace loaded ahead

template <typename T, bool BPTT>
__global__ void __launch_bounds__(kCeThreads) rate_ce_kernel(int64_t Tn, int64_t B, int C,
                                                             int pop, int64_t ld, int64_t Bn,
                                                             const T* spk, const int* labels,
                                                             float* loss, T* grad, double* terms,
                                                             int* ticket, const ReadoutBptt<T> r) {
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
  if constexpr (BPTT) {
    // neuron n of sample b is lane b*ld + n of every step
    for (int64_t n = threadIdx.x; n < ld; n += kCeThreads) {
      const float g = n < CP ? ccnt[n / pop] : 0.0f;
      const int64_t lane = b * ld + n;
      const float beta = __ldg(r.beta + (r.beta_col ? n : 0));
      const float thr = __ldg(r.thr + (r.thr_col ? n : 0));
      BwdLane st{0.0f, 0.0f, 0.0f, 0.0f, 0.0f};
      // chunks of kCeChunk steps from the last; the next chunk's loads are
      // issued before the current one is stepped (steps before 0 reload
      // step 0 and are not stepped)
      auto load_chunk = [&](int64_t tc, float (&u)[kCeChunk], uint32_t& zm) {
        zm = 0;
#pragma unroll
        for (int c = 0; c < kCeChunk; ++c) {
          const int64_t ts = tc - c >= 0 ? tc - c : 0;
          u[c] = Elem<T>::load1(r.mem + ts * step + lane);
          const uint32_t z = r.bits ? (__ldg(r.bits + ts * r.bits_row + (lane >> 3)) >> (lane & 7)) & 1u
                                    : (Elem<T>::load1(spk + ts * step + lane) != 0.0f ? 1u : 0u);
          zm |= z << c;
        }
      };
      float ucur[kCeChunk], unext[kCeChunk];
      uint32_t zcur, znext = 0;
      load_chunk(Tn - 1, ucur, zcur);
      for (int64_t tc = Tn - 1; tc >= 0; tc -= kCeChunk) {
        if (tc - kCeChunk >= 0) load_chunk(tc - kCeChunk, unext, znext);
#pragma unroll
        for (int c = 0; c < kCeChunk; ++c) {
          const int64_t ts = tc - c;
          if (ts < 0) break;
          const float du = bwd_step<false, -1, -1>(r.sa, beta, thr, 0.0f, ts + 1 < Tn, ucur[c],
                                                   ((zcur >> c) & 1u) != 0, 0.0f, g, 0.0f, 0.0f, st);
          Elem<T>::store1(r.gI + ts * step + lane, du);
          if (grad) Elem<T>::store1(grad + ts * step + lane, g);
        }
#pragma unroll
        for (int c = 0; c < kCeChunk; ++c) ucur[c] = unext[c];
        zcur = znext;
      }
    }
  } else {
    T* grow = grad + b * ld;
    for (int64_t n = threadIdx.x; n < ld; n += kCeThreads) {
      const float g = n < CP ? ccnt[n / pop] : 0.0f;
      for (int64_t t = 0; t < Tn; ++t) Elem<T>::store1(grow + t * step + n, g);
    }
  }
  // the last block to finish adds the loss terms
  __threadfence();
  __syncthreads();
  if (threadIdx.x == 0) last = atomicAdd(ticket, 1) == (int)(B - 1);
  __syncthreads();
  if (!last) return;
  __threadfence();
  // fixed order: thread i adds terms i, i + 256, ... in turn, each warp
  // folds its lanes by halves, and thread 0 adds the warp sums in order
  __shared__ double wsum[kCeThreads / 32];
  double part = 0.0;
  for (int64_t q = threadIdx.x; q < B; q += kCeThreads) part += __ldcg(terms + q);
  for (int o = 16; o > 0; o >>= 1) part += __shfl_down_sync(0xffffffffu, part, o);
  if ((threadIdx.x & 31) == 0) wsum[threadIdx.x >> 5] = part;
  __syncthreads();
  if (threadIdx.x == 0) {
    double total = 0.0;
    for (int k = 0; k < kCeThreads / 32; ++k) total += wsum[k];
    loss[0] = (float)(total / (double)Bn);
    *ticket = 0;
  }
}

template <typename T, bool BPTT = false>
cudaError_t launch_ce(int64_t Tn, int64_t B, int C, int pop, int64_t ld, int64_t Bn,
                      const void* spk, const int* labels, float* loss, void* grad, double* terms,
                      int* ticket, cudaStream_t st, const ReadoutBptt<T>& r = ReadoutBptt<T>{}) {
  const size_t smem = (size_t)(C * pop + C) * sizeof(float);
  const void* k = (const void*)rate_ce_kernel<T, BPTT>;
  const cudaError_t e = ensure_smem(k, smem);
  if (e != cudaSuccess) return e;
  return launch_pdl(rate_ce_kernel<T, BPTT>, dim3((unsigned)B), dim3(kCeThreads), smem, st, Tn,
                    B, C, pop, ld, Bn, static_cast<const T*>(spk), labels, loss,
                    static_cast<T*>(grad), terms, ticket, r);
}

template <typename T>
cudaError_t launch_ce_bptt(const snn_scan_desc* d, int C, int pop, int64_t Bn, const void* spk,
                           const int* labels, const float* beta, const float* thr, int beta_col,
                           int thr_col, const void* mem, const void* bits, float* loss,
                           void* grad, void* gI, double* terms, int* ticket, cudaStream_t st) {
  ReadoutBptt<T> r{};
  r.sa.reset = d->reset;
  r.sa.detach = d->detach_reset != 0;
  r.sa.sg = d->surrogate;
  r.sa.rec = 0;
  if (d->surrogate == SNN_SG_FAST_SIGMOID) {
    r.sa.sg_a = d->sg_param;
    r.sa.sg_b = 0.0f;
  } else {  // the constants the scan kernels take
    r.sa.sg_a = (float)(0.5 * (double)d->sg_param);
    r.sa.sg_b = (float)(3.14159265358979323846 * 0.5 * (double)d->sg_param);
  }
  r.beta = beta;
  r.thr = thr;
  r.beta_col = beta_col;
  r.thr_col = thr_col;
  r.mem = static_cast<const T*>(mem);
  r.bits = static_cast<const unsigned char*>(bits);
  r.bits_row = ((d->B * d->N + 7) / 8 + 15) / 16 * 16;
  r.gI = static_cast<T*>(gI);
  return launch_ce<T, true>(d->T, d->B, C, pop, d->N, Bn, spk, labels, loss, grad, terms, ticket,
                            st, r);
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

extern "C" snn_status_t snn_rate_ce_leaky_bwd(const snn_scan_desc* d, int64_t C, int64_t pop,
                                              int64_t batch_total, const void* spk,
                                              const int32_t* labels, const float* beta,
                                              const float* thr, const void* mem,
                                              const float* ckpt, float* loss, void* grad_spk,
                                              void* grad_I, void* ws, size_t ws_bytes,
                                              snn_stream_t stream) {
  if (!d || d->T < 0 || d->B < 0 || d->B > INT_MAX || d->N < 1 || d->reserved0 != 0 ||
      d->reserved1 != 0)
    return SNN_ERR_INVALID_ARG;
  if (C < 1 || pop < 1 || C > snn::kMaxClasses || pop > snn::kCeMaxNeurons / C || d->N < C * pop)
    return SNN_ERR_INVALID_ARG;
  if (d->reset < SNN_RESET_SUBTRACT || d->reset > SNN_RESET_NONE) return SNN_ERR_INVALID_ARG;
  if (d->surrogate != SNN_SG_FAST_SIGMOID && d->surrogate != SNN_SG_ATAN) return SNN_ERR_INVALID_ARG;
  if (!(d->sg_param > 0.0f)) return SNN_ERR_INVALID_ARG;
  if (d->io_dtype != SNN_F32 && d->io_dtype != SNN_BF16 && d->io_dtype != SNN_F16)
    return SNN_ERR_INVALID_ARG;
  if (d->save != SNN_SAVE_MEM) return SNN_ERR_UNSUPPORTED;
  int beta_col = 0, thr_col = 0;
  auto col_mode = [](int32_t mode, int* col) {
    if (mode == SNN_P_SCALAR) { *col = 0; return true; }
    if (mode == SNN_P_PER_NEURON) { *col = 1; return true; }
    return false;
  };
  if (!col_mode(d->beta_mode, &beta_col) || !col_mode(d->thr_mode, &thr_col)) return SNN_ERR_UNSUPPORTED;
  const int64_t Bn = batch_total > 0 ? batch_total : (d->B > 0 ? d->B : 1);
  if (batch_total > 0 && batch_total < d->B) return SNN_ERR_INVALID_ARG;
  const bool work = d->T > 0 && d->B > 0;
  if (!loss || (work && (!spk || !labels || !beta || !thr || !mem || !grad_I)))
    return SNN_ERR_INVALID_ARG;
  auto al16 = [](const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; };
  if (!al16(spk) || !al16(mem) || !al16(grad_I) || !al16(grad_spk) || !al16(ckpt) || !al16(ws))
    return SNN_ERR_ALIGNMENT;
  if (!ws || ws_bytes < snn_rate_ce_workspace_bytes(d->B)) return SNN_ERR_WORKSPACE;
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  if (d->B == 0)
    return cudaMemsetAsync(loss, 0, sizeof(float), st) == cudaSuccess ? SNN_OK : SNN_ERR_CUDA;
  unsigned char* w = static_cast<unsigned char*>(ws);
  int* ticket = reinterpret_cast<int*>(w);
  double* terms = reinterpret_cast<double*>(w + 256);
  cudaError_t e;
  switch (d->io_dtype) {
    case SNN_F32:
      e = snn::launch_ce_bptt<float>(d, (int)C, (int)pop, Bn, spk, labels, beta, thr, beta_col,
                                     thr_col, mem, ckpt, loss, grad_spk, grad_I, terms, ticket, st);
      break;
    case SNN_BF16:
      e = snn::launch_ce_bptt<__nv_bfloat16>(d, (int)C, (int)pop, Bn, spk, labels, beta, thr,
                                             beta_col, thr_col, mem, ckpt, loss, grad_spk, grad_I,
                                             terms, ticket, st);
      break;
    default:
      e = snn::launch_ce_bptt<__half>(d, (int)C, (int)pop, Bn, spk, labels, beta, thr, beta_col,
                                      thr_col, mem, ckpt, loss, grad_spk, grad_I, terms, ticket,
                                      st);
  }
  return e == cudaSuccess ? SNN_OK : SNN_ERR_CUDA;
}
