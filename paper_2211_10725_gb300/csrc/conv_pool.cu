// The convolutional SNN's layout kernels (Tab. I CSNN: 5x5 convolutions and
// 2x2 max pooling), for channel-last bf16 activations [M, H, W, C] with
// M = T*B.  A convolution runs as a tensor-core GEMM over patch rows:
//   im2col   cols[(m, oy, ox), (ky, kx, c)] = X[m, oy+ky, ox+kx, c]
//            (columns past KH*KW*Cin up to Kpad are zero), so the layer's
//            input current is cols * W^T with W [Cout, KH, KW, Cin];
//   col2im   dX[m, y, x, c] = sum over the (ky, kx) with a valid output
//            pixel (y-ky, x-kx) of dcols[(m, y-ky, x-kx), (ky, kx, c)],
//            added in (ky, kx) order in fp32 (deterministic);
//   max pool 2x2 windows, stride 2; the first maximum in window order
//            (row major) is kept and its position recorded, and the
//            backward routes the gradient there (every input element
//            belongs to one window, so no two threads write one element).
// With a channel count that is a multiple of 8 every kernel moves 8
// channels (16 bytes) per thread; otherwise one element per thread.
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include <climits>
#include <cstdint>

#include "launch.cuh"
#include "snn.h"

namespace snn {
namespace {

constexpr int kThreads = 256;

// Eight consecutive columns of one patch row per thread (one 16-byte store).
template <typename Ix>
__global__ void __launch_bounds__(kThreads) im2col_kernel(const __nv_bfloat16* __restrict__ X,
                                                          __nv_bfloat16* __restrict__ cols,
                                                          Ix rows, int H, int W, int Cin,
                                                          int KH, int KW, int Kpad) {
  grid_dep_wait();
  const int Ho = H - KH + 1, Wo = W - KW + 1;
  const int K = KH * KW * Cin;
  const int vec_per_row = Kpad / 8;
  const Ix i = (Ix)blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= rows * vec_per_row) return;
  const Ix r = i / vec_per_row;
  const int k0 = (int)(i - r * vec_per_row) * 8;
  const Ix m = r / (Ho * Wo);
  const int p = (int)(r - m * (Ho * Wo));
  const int oy = p / Wo, ox = p - oy * Wo;
  const __nv_bfloat16* xm = X + m * H * W * Cin;
  __align__(16) __nv_bfloat16 v[8];
#pragma unroll
  for (int j = 0; j < 8; ++j) {
    const int k = k0 + j;
    __nv_bfloat16 e = __float2bfloat16_rn(0.0f);
    if (k < K) {
      const int ky = k / (KW * Cin);
      const int rem = k - ky * KW * Cin;
      const int kx = rem / Cin, c = rem - kx * Cin;
      e = xm[((oy + ky) * W + (ox + kx)) * Cin + c];
    }
    v[j] = e;
  }
  *reinterpret_cast<uint4*>(cols + r * Kpad + k0) = *reinterpret_cast<const uint4*>(v);
}

template <typename Ix>
__global__ void __launch_bounds__(kThreads) col2im_kernel(const __nv_bfloat16* __restrict__ dcols,
                                                          __nv_bfloat16* __restrict__ dX,
                                                          Ix total, int H, int W, int Cin,
                                                          int KH, int KW, int Kpad) {
  grid_dep_wait();
  const int Ho = H - KH + 1, Wo = W - KW + 1;
  const Ix i = (Ix)blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= total) return;
  const int c = (int)(i % Cin);
  const Ix q = i / Cin;
  const int x = (int)(q % W);
  const Ix q2 = q / W;
  const int y = (int)(q2 % H);
  const Ix m = q2 / H;
  float s = 0.0f;
  for (int ky = 0; ky < KH; ++ky) {
    const int oy = y - ky;
    if (oy < 0 || oy >= Ho) continue;
    for (int kx = 0; kx < KW; ++kx) {
      const int ox = x - kx;
      if (ox < 0 || ox >= Wo) continue;
      const Ix r = (m * Ho + oy) * Wo + ox;
      s += __bfloat162float(dcols[r * Kpad + (ky * KW + kx) * Cin + c]);
    }
  }
  dX[i] = __float2bfloat16_rn(s);
}

template <typename Ix>
__global__ void __launch_bounds__(kThreads) maxpool_fwd_kernel(const __nv_bfloat16* __restrict__ X,
                                                               __nv_bfloat16* __restrict__ Y,
                                                               uint8_t* __restrict__ idx,
                                                               Ix total, int H, int W,
                                                               int C) {
  grid_dep_wait();
  const Ix i = (Ix)blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= total) return;
  const int Hp = H / 2, Wp = W / 2;
  const int c = (int)(i % C);
  const Ix q = i / C;
  const int px = (int)(q % Wp);
  const Ix q2 = q / Wp;
  const int py = (int)(q2 % Hp);
  const Ix m = q2 / Hp;
  const __nv_bfloat16* base = X + ((m * H + 2 * py) * W + 2 * px) * C + c;
  const Ix off[4] = {0, (Ix)C, (Ix)W * C, (Ix)W * C + C};
  float best = __bfloat162float(base[0]);
  int arg = 0;
#pragma unroll
  for (int j = 1; j < 4; ++j) {
    const float v = __bfloat162float(base[off[j]]);
    if (v > best) {  // strict: the first maximum is kept
      best = v;
      arg = j;
    }
  }
  Y[i] = __float2bfloat16_rn(best);
  idx[i] = (uint8_t)arg;
}

template <typename Ix>
__global__ void __launch_bounds__(kThreads) maxpool_bwd_kernel(const __nv_bfloat16* __restrict__ dY,
                                                               const uint8_t* __restrict__ idx,
                                                               __nv_bfloat16* __restrict__ dX,
                                                               Ix total, int H, int W,
                                                               int C) {
  grid_dep_wait();
  const Ix i = (Ix)blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= total) return;
  const int Hp = H / 2, Wp = W / 2;
  const int c = (int)(i % C);
  const Ix q = i / C;
  const int x = (int)(q % W);
  const Ix q2 = q / W;
  const int y = (int)(q2 % H);
  const Ix m = q2 / H;
  const Ix o = ((m * Hp + y / 2) * Wp + x / 2) * C + c;
  const int pos = (y & 1) * 2 + (x & 1);
  dX[i] = idx[o] == pos ? dY[o] : __float2bfloat16_rn(0.0f);
}

// ---- 8 channels per thread (C % 8 == 0, 16-byte aligned tensors) --------

union Pack8 {
  uint4 u;
  __nv_bfloat16 h[8];
};

// Thread i copies column group j = i % (Kpad/8) of patch row i / (Kpad/8):
// the 8 channels of one tap (groups past K are zero).
template <typename Ix>
__global__ void __launch_bounds__(kThreads) im2col_vec8_kernel(const uint4* __restrict__ X,
                                                               uint4* __restrict__ cols,
                                                               Ix rows, int H, int W, int Cin,
                                                               int KH, int KW, int Kpad) {
  grid_dep_wait();
  const int Ho = H - KH + 1, Wo = W - KW + 1;
  const int G = Cin / 8;  // channel groups per tap
  const int vpr = Kpad / 8;
  const Ix i = (Ix)blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= rows * vpr) return;
  const Ix r = i / vpr;
  const int j = (int)(i - r * vpr);
  uint4 v = make_uint4(0u, 0u, 0u, 0u);
  if (j < KH * KW * G) {
    const Ix m = r / (Ho * Wo);
    const int p = (int)(r - m * (Ho * Wo));
    const int oy = p / Wo, ox = p - oy * Wo;
    const int tap = j / G, g = j - tap * G;
    const int ky = tap / KW, kx = tap - ky * KW;
    v = X[((m * H + oy + ky) * W + ox + kx) * G + g];
  }
  cols[i] = v;
}

// As im2col_vec8_kernel, kIm2colPer vectors per thread (a block's threads
// stride over consecutive vectors, so stores stay coalesced and each thread
// has several loads in flight), the tap of each column group read from a
// shared-memory table instead of being divided out per element.
constexpr int kIm2colPer = 4;
constexpr int kIm2colMaxGroups = 4096;  // column groups (Kpad / 8) the table holds

template <typename Ix>
__global__ void __launch_bounds__(kThreads) im2col_vec8_multi_kernel(const uint4* __restrict__ X,
                                                                     uint4* __restrict__ cols,
                                                                     Ix rows, int H, int W,
                                                                     int Cin, int KH, int KW,
                                                                     int Kpad) {
  __shared__ int toff[kIm2colMaxGroups];  // input offset (16-byte units) of group j's tap, or -1
  const int Ho = H - KH + 1, Wo = W - KW + 1;
  const int G = Cin / 8;
  const int vpr = Kpad / 8;
  for (int j = threadIdx.x; j < vpr; j += blockDim.x) {
    int t = -1;
    if (j < KH * KW * G) {
      const int tap = j / G, g = j - tap * G;
      const int ky = tap / KW, kx = tap - ky * KW;
      t = (ky * W + kx) * G + g;
    }
    toff[j] = t;
  }
  __syncthreads();
  grid_dep_wait();
  const Ix total = rows * vpr;
  const Ix base = (Ix)blockIdx.x * blockDim.x * kIm2colPer + threadIdx.x;
  uint4 v[kIm2colPer];
#pragma unroll
  for (int u = 0; u < kIm2colPer; ++u) {
    const Ix i = base + (Ix)u * blockDim.x;
    v[u] = make_uint4(0u, 0u, 0u, 0u);
    if (i < total) {
      const Ix r = i / vpr;
      const int t = toff[(int)(i - r * vpr)];
      if (t >= 0) {
        const Ix m = r / (Ho * Wo);
        const int p = (int)(r - m * (Ho * Wo));
        const int oy = p / Wo, ox = p - oy * Wo;
        v[u] = X[((m * H + oy) * W + ox) * G + t];
      }
    }
  }
#pragma unroll
  for (int u = 0; u < kIm2colPer; ++u) {
    const Ix i = base + (Ix)u * blockDim.x;
    if (i < total) cols[i] = v[u];
  }
}

// Thread i sums the 8 channels of group i % G of pixel i / G over the taps
// that read it, in (ky, kx) order.
template <typename Ix, int KH_ = 0, int KW_ = 0>
__global__ void __launch_bounds__(kThreads) col2im_vec8_kernel(const uint4* __restrict__ dcols,
                                                               uint4* __restrict__ dX,
                                                               Ix total, int H, int W, int Cin,
                                                               int KH, int KW, int Kpad) {
  grid_dep_wait();
  const int Ho = H - KH + 1, Wo = W - KW + 1;
  const int G = Cin / 8, vpr = Kpad / 8;
  const Ix i = (Ix)blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= total) return;
  const Ix q = i / G;
  const int g = (int)(i - q * G);
  const int x = (int)(q % W);
  const Ix q2 = q / W;
  const int y = (int)(q2 % H);
  const Ix m = q2 / H;
  float s[8];
#pragma unroll
  for (int e = 0; e < 8; ++e) s[e] = 0.0f;
  if constexpr (KH_ > 0) {
    // fixed taps: one filter row's KW_ loads issued before its adds, which
    // still run in (ky, kx) order
#pragma unroll 1
    for (int ky = 0; ky < KH_; ++ky) {
      const int oy = y - ky;
      if (oy < 0 || oy >= Ho) continue;
      Pack8 v[KW_];
#pragma unroll
      for (int kx = 0; kx < KW_; ++kx) {
        const int ox = x - kx;
        v[kx].u = (ox >= 0 && ox < Wo) ? dcols[((m * Ho + oy) * Wo + ox) * vpr + (ky * KW_ + kx) * G + g]
                                       : make_uint4(0u, 0u, 0u, 0u);
      }
#pragma unroll
      for (int kx = 0; kx < KW_; ++kx) {
        const int ox = x - kx;
        if (ox >= 0 && ox < Wo) {
#pragma unroll
          for (int e = 0; e < 8; ++e) s[e] += __bfloat162float(v[kx].h[e]);
        }
      }
    }
  } else {
    for (int ky = 0; ky < KH; ++ky) {
      const int oy = y - ky;
      if (oy < 0 || oy >= Ho) continue;
      for (int kx = 0; kx < KW; ++kx) {
        const int ox = x - kx;
        if (ox < 0 || ox >= Wo) continue;
        const Ix r = (m * Ho + oy) * Wo + ox;
        Pack8 v;
        v.u = dcols[r * vpr + (ky * KW + kx) * G + g];
#pragma unroll
        for (int e = 0; e < 8; ++e) s[e] += __bfloat162float(v.h[e]);
      }
    }
  }
  Pack8 o;
#pragma unroll
  for (int e = 0; e < 8; ++e) o.h[e] = __float2bfloat16_rn(s[e]);
  dX[i] = o.u;
}

// Thread i pools the 8 channels of group i % G of output pixel i / G.
template <typename Ix>
__global__ void __launch_bounds__(kThreads) maxpool_fwd_vec8_kernel(const uint4* __restrict__ X,
                                                                    uint4* __restrict__ Y,
                                                                    uint2* __restrict__ idx,
                                                                    Ix total, int H, int W,
                                                                    int C) {
  grid_dep_wait();
  const Ix i = (Ix)blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= total) return;
  const int G = C / 8, Hp = H / 2, Wp = W / 2;
  const Ix q = i / G;
  const int g = (int)(i - q * G);
  const int px = (int)(q % Wp);
  const Ix q2 = q / Wp;
  const int py = (int)(q2 % Hp);
  const Ix m = q2 / Hp;
  const Ix base = ((m * H + 2 * py) * W + 2 * px) * G + g;
  Pack8 w[4];
  w[0].u = X[base];
  w[1].u = X[base + G];
  w[2].u = X[base + (Ix)W * G];
  w[3].u = X[base + (Ix)W * G + G];
  Pack8 best = w[0];
  uint8_t arg[8] = {0, 0, 0, 0, 0, 0, 0, 0};
#pragma unroll
  for (int j = 1; j < 4; ++j) {
#pragma unroll
    for (int e = 0; e < 8; ++e) {
      if (__bfloat162float(w[j].h[e]) > __bfloat162float(best.h[e])) {  // first maximum kept
        best.h[e] = w[j].h[e];
        arg[e] = (uint8_t)j;
      }
    }
  }
  Y[i] = best.u;
  uint2 a;
  a.x = (uint32_t)arg[0] | ((uint32_t)arg[1] << 8) | ((uint32_t)arg[2] << 16) | ((uint32_t)arg[3] << 24);
  a.y = (uint32_t)arg[4] | ((uint32_t)arg[5] << 8) | ((uint32_t)arg[6] << 16) | ((uint32_t)arg[7] << 24);
  idx[i] = a;
}

// Thread i routes the 8 channels of group i % G of output pixel i / G back
// to its window, writing all four positions (zero where not the maximum).
template <typename Ix>
__global__ void __launch_bounds__(kThreads) maxpool_bwd_vec8_kernel(const uint4* __restrict__ dY,
                                                                    const uint2* __restrict__ idx,
                                                                    uint4* __restrict__ dX,
                                                                    Ix total, int H, int W,
                                                                    int C) {
  grid_dep_wait();
  const Ix i = (Ix)blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= total) return;
  const int G = C / 8, Hp = H / 2, Wp = W / 2;
  const Ix q = i / G;
  const int g = (int)(i - q * G);
  const int px = (int)(q % Wp);
  const Ix q2 = q / Wp;
  const int py = (int)(q2 % Hp);
  const Ix m = q2 / Hp;
  Pack8 d;
  d.u = dY[i];
  const uint2 a = idx[i];
  const __nv_bfloat16 zero = __float2bfloat16_rn(0.0f);
  Pack8 o[4];
#pragma unroll
  for (int e = 0; e < 8; ++e) {
    const int pos = (int)(((e < 4 ? a.x : a.y) >> (8 * (e & 3))) & 0xFFu);
#pragma unroll
    for (int j = 0; j < 4; ++j) o[j].h[e] = pos == j ? d.h[e] : zero;
  }
  const Ix base = ((m * H + 2 * py) * W + 2 * px) * G + g;
  dX[base] = o[0].u;
  dX[base + G] = o[1].u;
  dX[base + (Ix)W * G] = o[2].u;
  dX[base + (Ix)W * G + G] = o[3].u;
}

bool aligned(const void* p, uintptr_t a) { return (reinterpret_cast<uintptr_t>(p) & (a - 1)) == 0; }

unsigned blocks_for(int64_t n) { return (unsigned)((n + kThreads - 1) / kThreads); }

}  // namespace
}  // namespace snn

using namespace snn;

extern "C" snn_status_t snn_im2col_nhwc(int64_t M, int64_t H, int64_t W, int64_t Cin, int64_t KH,
                                        int64_t KW, int64_t Kpad, const void* X, void* cols,
                                        snn_stream_t stream) {
  if (M < 0 || KH < 1 || KW < 1 || H < KH || W < KW || Cin < 1) return SNN_ERR_INVALID_ARG;
  if (H * W * Cin > INT_MAX / 2 || Kpad > INT_MAX / 2) return SNN_ERR_INVALID_ARG;
  if (Kpad < KH * KW * Cin || Kpad % 8 != 0) return SNN_ERR_INVALID_ARG;
  if (M == 0) return SNN_OK;
  if (!X || !cols) return SNN_ERR_INVALID_ARG;
  if (!aligned(cols, 16) || !aligned(X, 2)) return SNN_ERR_ALIGNMENT;
  const int64_t rows = M * (H - KH + 1) * (W - KW + 1);
  const int64_t n = rows * (Kpad / 8);
  if (n / kThreads >= INT_MAX) return SNN_ERR_INVALID_ARG;
  const bool i32 = rows * Kpad < INT_MAX && M * H * W * Cin < INT_MAX;  // 32-bit index math
  if (Cin % 8 == 0 && aligned(X, 16) && Kpad / 8 <= kIm2colMaxGroups) {
    const unsigned nb = (unsigned)((n + (int64_t)kThreads * kIm2colPer - 1) / ((int64_t)kThreads * kIm2colPer));
    const cudaError_t e =
        i32 ? launch_pdl(im2col_vec8_multi_kernel<int>, dim3(nb), dim3(kThreads), 0,
                         reinterpret_cast<cudaStream_t>(stream), static_cast<const uint4*>(X),
                         static_cast<uint4*>(cols), rows, (int)H, (int)W, (int)Cin, (int)KH,
                         (int)KW, (int)Kpad)
            : launch_pdl(im2col_vec8_multi_kernel<int64_t>, dim3(nb), dim3(kThreads), 0,
                         reinterpret_cast<cudaStream_t>(stream), static_cast<const uint4*>(X),
                         static_cast<uint4*>(cols), rows, (int)H, (int)W, (int)Cin, (int)KH,
                         (int)KW, (int)Kpad);
    return e == cudaSuccess ? SNN_OK : SNN_ERR_CUDA;
  }
  if (Cin % 8 == 0 && aligned(X, 16)) {
    const cudaError_t e = i32 ? launch_pdl(im2col_vec8_kernel<int>, dim3(blocks_for(n)), dim3(kThreads), 0,
                                     reinterpret_cast<cudaStream_t>(stream),
                                     static_cast<const uint4*>(X), static_cast<uint4*>(cols), rows,
                                     (int)H, (int)W, (int)Cin, (int)KH, (int)KW, (int)Kpad)
                                   : launch_pdl(im2col_vec8_kernel<int64_t>, dim3(blocks_for(n)), dim3(kThreads), 0,
                                     reinterpret_cast<cudaStream_t>(stream),
                                     static_cast<const uint4*>(X), static_cast<uint4*>(cols), rows,
                                     (int)H, (int)W, (int)Cin, (int)KH, (int)KW, (int)Kpad);
    return e == cudaSuccess ? SNN_OK : SNN_ERR_CUDA;
  }
  const cudaError_t e = i32 ? launch_pdl(im2col_kernel<int>, dim3(blocks_for(n)), dim3(kThreads), 0,
                                   reinterpret_cast<cudaStream_t>(stream),
                                   static_cast<const __nv_bfloat16*>(X),
                                   static_cast<__nv_bfloat16*>(cols), rows, (int)H, (int)W, (int)Cin,
                                   (int)KH, (int)KW, (int)Kpad)
                                   : launch_pdl(im2col_kernel<int64_t>, dim3(blocks_for(n)), dim3(kThreads), 0,
                                   reinterpret_cast<cudaStream_t>(stream),
                                   static_cast<const __nv_bfloat16*>(X),
                                   static_cast<__nv_bfloat16*>(cols), rows, (int)H, (int)W, (int)Cin,
                                   (int)KH, (int)KW, (int)Kpad);
  return e == cudaSuccess ? SNN_OK : SNN_ERR_CUDA;
}

extern "C" snn_status_t snn_col2im_nhwc(int64_t M, int64_t H, int64_t W, int64_t Cin, int64_t KH,
                                        int64_t KW, int64_t Kpad, const void* dcols, void* dX,
                                        snn_stream_t stream) {
  if (M < 0 || KH < 1 || KW < 1 || H < KH || W < KW || Cin < 1) return SNN_ERR_INVALID_ARG;
  if (H * W * Cin > INT_MAX / 2 || Kpad > INT_MAX / 2) return SNN_ERR_INVALID_ARG;
  if (Kpad < KH * KW * Cin) return SNN_ERR_INVALID_ARG;
  if (M == 0) return SNN_OK;
  if (!dcols || !dX) return SNN_ERR_INVALID_ARG;
  if (!aligned(dcols, 2) || !aligned(dX, 2)) return SNN_ERR_ALIGNMENT;
  const int64_t n = M * H * W * Cin;
  if (n / kThreads >= INT_MAX) return SNN_ERR_INVALID_ARG;
  const bool i32 = M * (H - KH + 1) * (W - KW + 1) * Kpad < INT_MAX && n < INT_MAX;
  if (Cin % 8 == 0 && Kpad % 8 == 0 && aligned(dcols, 16) && aligned(dX, 16)) {
    cudaError_t e;
    if (KH == 5 && KW == 5 && i32)
      e = launch_pdl(col2im_vec8_kernel<int, 5, 5>, dim3(blocks_for(n / 8)), dim3(kThreads), 0,
                     reinterpret_cast<cudaStream_t>(stream), static_cast<const uint4*>(dcols),
                     static_cast<uint4*>(dX), n / 8, (int)H, (int)W, (int)Cin, (int)KH, (int)KW,
                     (int)Kpad);
    else
      e = i32 ? launch_pdl(col2im_vec8_kernel<int>, dim3(blocks_for(n / 8)), dim3(kThreads), 0,
                                     reinterpret_cast<cudaStream_t>(stream),
                                     static_cast<const uint4*>(dcols), static_cast<uint4*>(dX),
                                     n / 8, (int)H, (int)W, (int)Cin, (int)KH, (int)KW, (int)Kpad)
                                   : launch_pdl(col2im_vec8_kernel<int64_t>, dim3(blocks_for(n / 8)), dim3(kThreads), 0,
                                     reinterpret_cast<cudaStream_t>(stream),
                                     static_cast<const uint4*>(dcols), static_cast<uint4*>(dX),
                                     n / 8, (int)H, (int)W, (int)Cin, (int)KH, (int)KW, (int)Kpad);
    return e == cudaSuccess ? SNN_OK : SNN_ERR_CUDA;
  }
  const cudaError_t e = i32 ? launch_pdl(col2im_kernel<int>, dim3(blocks_for(n)), dim3(kThreads), 0,
                                   reinterpret_cast<cudaStream_t>(stream),
                                   static_cast<const __nv_bfloat16*>(dcols),
                                   static_cast<__nv_bfloat16*>(dX), n, (int)H, (int)W, (int)Cin,
                                   (int)KH, (int)KW, (int)Kpad)
                                   : launch_pdl(col2im_kernel<int64_t>, dim3(blocks_for(n)), dim3(kThreads), 0,
                                   reinterpret_cast<cudaStream_t>(stream),
                                   static_cast<const __nv_bfloat16*>(dcols),
                                   static_cast<__nv_bfloat16*>(dX), n, (int)H, (int)W, (int)Cin,
                                   (int)KH, (int)KW, (int)Kpad);
  return e == cudaSuccess ? SNN_OK : SNN_ERR_CUDA;
}

extern "C" snn_status_t snn_maxpool2_fwd_nhwc(int64_t M, int64_t H, int64_t W, int64_t C,
                                              const void* X, void* Y, uint8_t* idx,
                                              snn_stream_t stream) {
  if (M < 0 || H < 2 || W < 2 || C < 1 || H % 2 || W % 2) return SNN_ERR_INVALID_ARG;
  if (H * W * C > INT_MAX / 2) return SNN_ERR_INVALID_ARG;
  if (M == 0) return SNN_OK;
  if (!X || !Y || !idx) return SNN_ERR_INVALID_ARG;
  if (!aligned(X, 2) || !aligned(Y, 2)) return SNN_ERR_ALIGNMENT;
  const int64_t n = M * (H / 2) * (W / 2) * C;
  if (n / kThreads >= INT_MAX) return SNN_ERR_INVALID_ARG;
  const bool i32 = M * H * W * C < INT_MAX;
  if (C % 8 == 0 && aligned(X, 16) && aligned(Y, 16) && aligned(idx, 8)) {
    const cudaError_t e = i32 ? launch_pdl(maxpool_fwd_vec8_kernel<int>, dim3(blocks_for(n / 8)),
                                     dim3(kThreads), 0, reinterpret_cast<cudaStream_t>(stream),
                                     static_cast<const uint4*>(X), static_cast<uint4*>(Y),
                                     reinterpret_cast<uint2*>(idx), n / 8, (int)H, (int)W, (int)C)
                                   : launch_pdl(maxpool_fwd_vec8_kernel<int64_t>, dim3(blocks_for(n / 8)),
                                     dim3(kThreads), 0, reinterpret_cast<cudaStream_t>(stream),
                                     static_cast<const uint4*>(X), static_cast<uint4*>(Y),
                                     reinterpret_cast<uint2*>(idx), n / 8, (int)H, (int)W, (int)C);
    return e == cudaSuccess ? SNN_OK : SNN_ERR_CUDA;
  }
  const cudaError_t e = i32 ? launch_pdl(maxpool_fwd_kernel<int>, dim3(blocks_for(n)), dim3(kThreads), 0,
                                   reinterpret_cast<cudaStream_t>(stream),
                                   static_cast<const __nv_bfloat16*>(X),
                                   static_cast<__nv_bfloat16*>(Y), idx, n, (int)H, (int)W, (int)C)
                                   : launch_pdl(maxpool_fwd_kernel<int64_t>, dim3(blocks_for(n)), dim3(kThreads), 0,
                                   reinterpret_cast<cudaStream_t>(stream),
                                   static_cast<const __nv_bfloat16*>(X),
                                   static_cast<__nv_bfloat16*>(Y), idx, n, (int)H, (int)W, (int)C);
  return e == cudaSuccess ? SNN_OK : SNN_ERR_CUDA;
}

extern "C" snn_status_t snn_maxpool2_bwd_nhwc(int64_t M, int64_t H, int64_t W, int64_t C,
                                              const void* dY, const uint8_t* idx, void* dX,
                                              snn_stream_t stream) {
  if (M < 0 || H < 2 || W < 2 || C < 1 || H % 2 || W % 2) return SNN_ERR_INVALID_ARG;
  if (H * W * C > INT_MAX / 2) return SNN_ERR_INVALID_ARG;
  if (M == 0) return SNN_OK;
  if (!dY || !idx || !dX) return SNN_ERR_INVALID_ARG;
  if (!aligned(dY, 2) || !aligned(dX, 2)) return SNN_ERR_ALIGNMENT;
  const int64_t n = M * H * W * C;
  if (n / kThreads >= INT_MAX) return SNN_ERR_INVALID_ARG;
  const bool i32 = n < INT_MAX;
  if (C % 8 == 0 && aligned(dY, 16) && aligned(dX, 16) && aligned(idx, 8)) {
    const int64_t np = n / 32;  // output pixels x channel groups
    const cudaError_t e = i32 ? launch_pdl(maxpool_bwd_vec8_kernel<int>, dim3(blocks_for(np)),
                                     dim3(kThreads), 0, reinterpret_cast<cudaStream_t>(stream),
                                     static_cast<const uint4*>(dY),
                                     reinterpret_cast<const uint2*>(idx), static_cast<uint4*>(dX),
                                     np, (int)H, (int)W, (int)C)
                                   : launch_pdl(maxpool_bwd_vec8_kernel<int64_t>, dim3(blocks_for(np)),
                                     dim3(kThreads), 0, reinterpret_cast<cudaStream_t>(stream),
                                     static_cast<const uint4*>(dY),
                                     reinterpret_cast<const uint2*>(idx), static_cast<uint4*>(dX),
                                     np, (int)H, (int)W, (int)C);
    return e == cudaSuccess ? SNN_OK : SNN_ERR_CUDA;
  }
  const cudaError_t e = i32 ? launch_pdl(maxpool_bwd_kernel<int>, dim3(blocks_for(n)), dim3(kThreads), 0,
                                   reinterpret_cast<cudaStream_t>(stream),
                                   static_cast<const __nv_bfloat16*>(dY), idx,
                                   static_cast<__nv_bfloat16*>(dX), n, (int)H, (int)W, (int)C)
                                   : launch_pdl(maxpool_bwd_kernel<int64_t>, dim3(blocks_for(n)), dim3(kThreads), 0,
                                   reinterpret_cast<cudaStream_t>(stream),
                                   static_cast<const __nv_bfloat16*>(dY), idx,
                                   static_cast<__nv_bfloat16*>(dX), n, (int)H, (int)W, (int)C);
  return e == cudaSuccess ? SNN_OK : SNN_ERR_CUDA;
}
