// Convolution with few input channels (the CSNN's first layer, Tab. I:
// 5x5 filters over a 1-channel 28x28 map) on the CUDA cores.  Each output
// pixel needs KH*KW*Cin <= 32 products per channel, so a patch-row GEMM
// would move 2*Kpad bytes of patch per output pixel for so little
// arithmetic; here each image is staged once in shared memory instead.
//
//   forward   I[m, oy, ox, o] = sum_k X[m, oy+ky, ox+kx, c] * W[o, k]
//             k = (ky*KW + kx)*Cin + c, fp32 fused multiply-adds in k order
//   weight    dW[o, k] = sum over (m, oy, ox) of dI[m, oy, ox, o] *
//   gradient  X[m, oy+ky, ox+kx, c]; block b sums images b, b + G, ... in
//             order, lanes add their pixels in order, and the warp trees
//             and the final sum over the G block partials (strided lane sums,
//             then a shuffle tree) run in a fixed order, so the result is
//             the same on every call.
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include <climits>
#include <cstdint>

#include "launch.cuh"
#include "snn.h"

namespace snn {
namespace {

constexpr int kMaxK = 32;      // KH*KW*Cin
constexpr int kMaxCout = 16;   // output channels (weights padded to 16 in shared memory)
constexpr int kMaxImage = 8192;  // H*W*Cin elements staged per image (32 KB)
constexpr int kDwThreads = 128;  // 4 warps: warp w owns output channels 4w .. 4w+3
constexpr int kDwBlocks = 304;   // fixed block count of the weight gradient (2 per SM of 152)

// Window taps: compile-time when KH_ > 0 (the 5x5 and 3x3 single-channel
// cases, offsets ky*W + kx folded into the loads), else read from soff.
template <int KH_, int KW_, int CIN_>
struct Taps {
  static constexpr bool kFixed = KH_ > 0;
  static constexpr int kK = KH_ * KW_ * CIN_;
};

// Prefetch of one image's input map into registers (16-byte vectors,
// kPreVec per thread) while the previous image is being used.
constexpr int kPreVec = 4;

__device__ __forceinline__ void unpack8(const uint4& u, float* dst) {
  const __nv_bfloat162* h = reinterpret_cast<const __nv_bfloat162*>(&u);
#pragma unroll
  for (int j = 0; j < 4; ++j) {
    const float2 f = __bfloat1622float2(h[j]);
    dst[2 * j] = f.x;
    dst[2 * j + 1] = f.y;
  }
}

// Forward: persistent blocks over images; the image is staged in shared
// memory as fp32 (the next one's 16-byte vectors in flight in registers),
// weights as [k][16] fp32.  Thread u of an image computes output pixels
// 2*(u / CG) and 2*(u / CG) + 1 (horizontally adjacent) for channels
// 4*(u % CG) .. +3 (CG = Cout/4 channel groups) with paired fp32 FMAs (two
// independent round-to-nearest FMAs per instruction), so the CG threads of
// a pixel pair store one contiguous 2*Cout*4-byte run.
template <int KH_, int KW_, int CIN_>
__global__ void __launch_bounds__(256) conv_small_fwd_kernel(
    const __nv_bfloat16* __restrict__ X, const __nv_bfloat16* __restrict__ Wt,
    float* __restrict__ I, int64_t M, int H, int W, int Cin, int Cout, int KH, int KW, int ldw,
    int vec) {
  __shared__ __align__(16) float sw[kMaxK * kMaxCout];  // [k][16]
  __shared__ int soff[kMaxK];
  extern __shared__ __align__(16) float sx[];  // the image, H*W*Cin
  using Tp = Taps<KH_, KW_, CIN_>;
  const int K = Tp::kFixed ? Tp::kK : KH * KW * Cin;
  const int Ho = H - (Tp::kFixed ? KH_ : KH) + 1, Wo = W - (Tp::kFixed ? KW_ : KW) + 1;
  const int P = Ho * Wo;
  const int img = H * W * Cin;
  const int nv = vec ? img / 8 : 0;
  const int Wo2 = (Wo + 1) / 2;  // pixel pairs per output row
  const int CG = Cout / 4;
  const int units = Ho * Wo2 * CG;
  grid_dep_wait();
  for (int e = threadIdx.x; e < kMaxK * kMaxCout; e += blockDim.x) {
    const int k = e / kMaxCout, o = e - k * kMaxCout;
    sw[e] = (k < K && o < Cout) ? __bfloat162float(Wt[(int64_t)o * ldw + k]) : 0.0f;
  }
  for (int k = threadIdx.x; k < K; k += blockDim.x) {
    const int tap = k / Cin, c = k - tap * Cin;
    const int ky = tap / KW, kx = tap - ky * KW;
    soff[k] = (ky * W + kx) * Cin + c;
  }
  uint4 pre[kPreVec];
  auto fetch = [&](int64_t m) {
    const uint4* src = reinterpret_cast<const uint4*>(X + m * img);
#pragma unroll
    for (int j = 0; j < kPreVec; ++j) {
      const int v = threadIdx.x + j * blockDim.x;
      if (v < nv) pre[j] = src[v];
    }
  };
  if (vec && (int64_t)blockIdx.x < M) fetch(blockIdx.x);
  for (int64_t m = blockIdx.x; m < M; m += gridDim.x) {
    __syncthreads();  // the previous image is no longer read
    if (vec) {
#pragma unroll
      for (int j = 0; j < kPreVec; ++j) {
        const int v = threadIdx.x + j * blockDim.x;
        if (v < nv) unpack8(pre[j], sx + 8 * v);
      }
    } else {
      const __nv_bfloat16* xm = X + m * img;
      for (int e = threadIdx.x; e < img; e += blockDim.x) sx[e] = __bfloat162float(xm[e]);
    }
    __syncthreads();
    if (vec && m + gridDim.x < M) fetch(m + gridDim.x);
    for (int u = threadIdx.x; u < units; u += blockDim.x) {
      const int pp = u / CG, cg = u - pp * CG;
      const int oy = pp / Wo2, ox = 2 * (pp - oy * Wo2);
      const bool two = ox + 1 < Wo;
      const int base = (oy * W + ox) * Cin;
      float2 a0l = make_float2(0.0f, 0.0f), a0h = a0l, a1l = a0l, a1h = a0l;
      const float* wc = sw + 4 * cg;
      auto tap = [&](int k, int off) {
        const float x0 = sx[base + off];
        const float x1 = two ? sx[base + off + Cin] : 0.0f;
        const float4 w4 = *reinterpret_cast<const float4*>(wc + k * kMaxCout);
        const float2 wl = make_float2(w4.x, w4.y), wh = make_float2(w4.z, w4.w);
        const float2 x0p = make_float2(x0, x0), x1p = make_float2(x1, x1);
        a0l = __ffma2_rn(x0p, wl, a0l);
        a0h = __ffma2_rn(x0p, wh, a0h);
        a1l = __ffma2_rn(x1p, wl, a1l);
        a1h = __ffma2_rn(x1p, wh, a1h);
      };
      if constexpr (Tp::kFixed) {
#pragma unroll
        for (int ky = 0; ky < KH_; ++ky)
#pragma unroll
          for (int kx = 0; kx < KW_; ++kx)
#pragma unroll
            for (int c = 0; c < CIN_; ++c) tap((ky * KW_ + kx) * CIN_ + c, (ky * W + kx) * CIN_ + c);
      } else {
        for (int k = 0; k < K; ++k) tap(k, soff[k]);
      }
      float* d0 = I + (m * P + oy * Wo + ox) * Cout + 4 * cg;
      *reinterpret_cast<float4*>(d0) = make_float4(a0l.x, a0l.y, a0h.x, a0h.y);
      if (two) *reinterpret_cast<float4*>(d0 + Cout) = make_float4(a1l.x, a1l.y, a1h.x, a1h.y);
    }
  }
}

__device__ __forceinline__ void cp_async16(void* dst, const void* src) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(
                   static_cast<uint32_t>(__cvta_generic_to_shared(dst))),
               "l"(src)
               : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
__device__ __forceinline__ void cp_async_wait_all_but_one() {
  asm volatile("cp.async.wait_group 1;" ::: "memory");
}

// Weight gradient: block b takes images b, b + G, ... (G fixed).  Each
// image's input map and output gradient are copied raw (bf16, cp.async,
// double-buffered: the next image's copies are in flight while this one is
// summed), then expanded in shared memory to fp32: the map as is, the
// gradient transposed to [o][p] so that lanes over pixels read it without
// bank conflicts.  Warp w owns output channels 4w .. 4w+3 and all K taps (2
// x KC paired accumulators per lane); lane l takes pixels l, l + 32, ... At
// the end each warp adds its lanes in a fixed shuffle tree and writes the
// block's partial.
template <int KH_, int KW_, int CIN_, int KC>
__global__ void __launch_bounds__(kDwThreads) conv_small_dw_kernel(
    const __nv_bfloat16* __restrict__ X, const __nv_bfloat16* __restrict__ dI,
    float* __restrict__ part, int64_t M, int H, int W, int Cin, int Cout, int KH, int KW,
    int vec) {
  __shared__ int soff[kMaxK];
  extern __shared__ __align__(16) unsigned char dsm[];
  using Tp = Taps<KH_, KW_, CIN_>;
  const int K = Tp::kFixed ? Tp::kK : KH * KW * Cin;
  const int Ho = H - (Tp::kFixed ? KH_ : KH) + 1, Wo = W - (Tp::kFixed ? KW_ : KW) + 1;
  const int P = Ho * Wo;
  const int img = H * W * Cin;
  const int pix = P * Cout;
  const int rx = (img * 2 + 15) & ~15, rd = (pix * 2 + 15) & ~15;  // raw bytes
  auto raw = [&](int b) { return dsm + b * (rx + rd); };  // two raw buffers
  float* sx = reinterpret_cast<float*>(dsm + 2 * (rx + rd));       // [img]
  float* sdT = sx + ((img + 3) & ~3);                               // [Cout][P]
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int o0 = 4 * warp;
  const int64_t G = gridDim.x;
  grid_dep_wait();
  for (int k = threadIdx.x; k < K; k += blockDim.x) {
    const int tap = k / Cin, c = k - tap * Cin;
    const int ky = tap / KW, kx = tap - ky * KW;
    soff[k] = (ky * W + kx) * Cin + c;
  }
  auto stage = [&](int64_t m, int b) {
    if (vec) {
      const unsigned char* gx = reinterpret_cast<const unsigned char*>(X + m * img);
      const unsigned char* gd = reinterpret_cast<const unsigned char*>(dI + m * pix);
      for (int c = threadIdx.x; c < img / 8; c += blockDim.x) cp_async16(raw(b) + 16 * c, gx + 16 * c);
      for (int c = threadIdx.x; c < pix / 8; c += blockDim.x)
        cp_async16(raw(b) + rx + 16 * c, gd + 16 * c);
    } else {
      __nv_bfloat16* hx = reinterpret_cast<__nv_bfloat16*>(raw(b));
      __nv_bfloat16* hd = reinterpret_cast<__nv_bfloat16*>(raw(b) + rx);
      for (int e = threadIdx.x; e < img; e += blockDim.x) hx[e] = X[m * img + e];
      for (int e = threadIdx.x; e < pix; e += blockDim.x) hd[e] = dI[m * pix + e];
    }
    cp_async_commit();
  };
  float2 acc[2][KC];  // [channel pair][tap]: (o0 + 2j, o0 + 2j + 1)
#pragma unroll
  for (int j = 0; j < 2; ++j)
#pragma unroll
    for (int k = 0; k < KC; ++k) acc[j][k] = make_float2(0.0f, 0.0f);
  // two copy groups in flight before the loop, one more per image: image i
  // of this block is group i, complete once at most one newer group pends
  if ((int64_t)blockIdx.x < M) stage(blockIdx.x, 0);
  else cp_async_commit();
  if ((int64_t)blockIdx.x + G < M) stage(blockIdx.x + G, 1);
  else cp_async_commit();
  int i = 0;
  for (int64_t m = blockIdx.x; m < M; m += G, ++i) {
    const int b = i & 1;
    cp_async_wait_all_but_one();  // image m's copies have landed (m + G may be in flight)
    __syncthreads();              // for every thread; the fp32 buffers are free
    const __nv_bfloat16* hx = reinterpret_cast<const __nv_bfloat16*>(raw(b));
    const __nv_bfloat16* hd = reinterpret_cast<const __nv_bfloat16*>(raw(b) + rx);
    if (vec) {
      // 8 channels of one pixel per 16-byte vector (Cout is a multiple of 8 here)
      const int gpp = Cout / 8;
      for (int v = threadIdx.x; v < img / 8; v += blockDim.x)
        unpack8(reinterpret_cast<const uint4*>(hx)[v], sx + 8 * v);
      for (int v = threadIdx.x; v < pix / 8; v += blockDim.x) {
        const int p = v / gpp, o = (v - p * gpp) * 8;
        float f[8];
        unpack8(reinterpret_cast<const uint4*>(hd)[v], f);
#pragma unroll
        for (int j = 0; j < 8; ++j) sdT[(o + j) * P + p] = f[j];
      }
    } else {
      for (int e = threadIdx.x; e < img; e += blockDim.x) sx[e] = __bfloat162float(hx[e]);
      for (int e = threadIdx.x; e < pix; e += blockDim.x) {
        const int p = e / Cout, o = e - p * Cout;
        sdT[o * P + p] = __bfloat162float(hd[e]);
      }
    }
    __syncthreads();  // raw buffer b is free again
    if (m + 2 * G < M) stage(m + 2 * G, b);
    else cp_async_commit();  // an empty group keeps the wait count uniform
    if (o0 < Cout) {
      const float* g0 = sdT + (o0 + 0) * P;
      const float* g1 = sdT + (o0 + 1) * P;
      const float* g2 = sdT + (o0 + 2) * P;
      const float* g3 = sdT + (o0 + 3) * P;
      for (int p = lane; p < P; p += 32) {
        const int oy = p / Wo, ox = p - oy * Wo;
        const float* xb = sx + (oy * W + ox) * Cin;
        const float2 ga = make_float2(g0[p], g1[p]), gb = make_float2(g2[p], g3[p]);
        if constexpr (Tp::kFixed) {
#pragma unroll
          for (int ky = 0; ky < KH_; ++ky)
#pragma unroll
            for (int kx = 0; kx < KW_; ++kx)
#pragma unroll
              for (int c = 0; c < CIN_; ++c) {
                const int k = (ky * KW_ + kx) * CIN_ + c;
                const float xv = xb[(ky * W + kx) * CIN_ + c];
                const float2 xp = make_float2(xv, xv);
                acc[0][k] = __ffma2_rn(ga, xp, acc[0][k]);
                acc[1][k] = __ffma2_rn(gb, xp, acc[1][k]);
              }
        } else {
#pragma unroll
          for (int k = 0; k < KC; ++k) {
            if (k < K) {
              const float xv = xb[soff[k]];
              const float2 xp = make_float2(xv, xv);
              acc[0][k] = __ffma2_rn(ga, xp, acc[0][k]);
              acc[1][k] = __ffma2_rn(gb, xp, acc[1][k]);
            }
          }
        }
      }
    }
  }
  // lanes' sums in a fixed tree; lane 0 writes the block's partial
#pragma unroll
  for (int j = 0; j < 2; ++j)
#pragma unroll
    for (int k = 0; k < KC; ++k) {
      float2 v = acc[j][k];
#pragma unroll
      for (int s = 16; s > 0; s >>= 1) {
        v.x += __shfl_xor_sync(0xffffffffu, v.x, s);
        v.y += __shfl_xor_sync(0xffffffffu, v.y, s);
      }
      acc[j][k] = v;
    }
  if (lane == 0 && o0 < Cout) {
    float* pb = part + (int64_t)blockIdx.x * Cout * K;
#pragma unroll
    for (int k = 0; k < KC; ++k)
      if (k < K) {
        pb[(o0 + 0) * K + k] = acc[0][k].x;
        pb[(o0 + 1) * K + k] = acc[0][k].y;
        pb[(o0 + 2) * K + k] = acc[1][k].x;
        pb[(o0 + 3) * K + k] = acc[1][k].y;
      }
  }
}

// ---- Single input channel, fixed KH x KW: sliding windows --------------
//
// Thread t of an image owns output row oy = t / CG and channel pair cg =
// t % CG (channels 2cg, 2cg+1; CG = Cout/2) and walks the row left to
// right, keeping the KH x KW input window in registers: each step shifts it
// one column and loads the KH new values, so shared memory is read once per
// input value and row.  Two channels per thread keep the register count
// near 100, so that about 18 warps fit on an SM.

constexpr int kSlideMaxThreads = 512;

template <int KH_, int KW_>
__global__ void __launch_bounds__(kSlideMaxThreads) conv_slide_fwd_kernel(
    const __nv_bfloat16* __restrict__ X, const __nv_bfloat16* __restrict__ Wt,
    float* __restrict__ I, int64_t M, int H, int W, int Cout, int ldw, int vec) {
  constexpr int KK = KH_ * KW_;
  extern __shared__ __align__(16) float sx[];  // the image, H*W
  const int Ho = H - KH_ + 1, Wo = W - KW_ + 1, P = Ho * Wo;
  const int img = H * W;
  const int nv = vec ? img / 8 : 0;
  const int CG = Cout / 2;
  const int t = threadIdx.x;
  const bool active = t < Ho * CG;
  const int oy = t / CG, cg = t - (t / CG) * CG;
  grid_dep_wait();
  float2 w2[KK];  // this thread's 2 channels of every tap
#pragma unroll
  for (int k = 0; k < KK; ++k)
    w2[k] = active ? make_float2(__bfloat162float(Wt[(int64_t)(2 * cg) * ldw + k]),
                                 __bfloat162float(Wt[(int64_t)(2 * cg + 1) * ldw + k]))
                   : make_float2(0.0f, 0.0f);
  uint4 pre[kPreVec];
  auto fetch = [&](int64_t m) {
    const uint4* src = reinterpret_cast<const uint4*>(X + m * img);
#pragma unroll
    for (int j = 0; j < kPreVec; ++j) {
      const int v = t + j * blockDim.x;
      if (v < nv) pre[j] = src[v];
    }
  };
  if (vec && (int64_t)blockIdx.x < M) fetch(blockIdx.x);
  for (int64_t m = blockIdx.x; m < M; m += gridDim.x) {
    __syncthreads();  // the previous image is no longer read
    if (vec) {
#pragma unroll
      for (int j = 0; j < kPreVec; ++j) {
        const int v = t + j * blockDim.x;
        if (v < nv) unpack8(pre[j], sx + 8 * v);
      }
    } else {
      for (int e = t; e < img; e += blockDim.x) sx[e] = __bfloat162float(X[m * img + e]);
    }
    __syncthreads();
    if (vec && m + gridDim.x < M) fetch(m + gridDim.x);
    if (!active) continue;
    const float* row = sx + oy * W;
    float win[KH_][KW_];
#pragma unroll
    for (int ky = 0; ky < KH_; ++ky)
#pragma unroll
      for (int kx = 1; kx < KW_; ++kx) win[ky][kx] = row[ky * W + kx - 1];
    float* out = I + (m * P + (int64_t)oy * Wo) * Cout + 2 * cg;
#pragma unroll 2
    for (int ox = 0; ox < Wo; ++ox) {
#pragma unroll
      for (int ky = 0; ky < KH_; ++ky) {
#pragma unroll
        for (int kx = 0; kx < KW_ - 1; ++kx) win[ky][kx] = win[ky][kx + 1];
        win[ky][KW_ - 1] = row[ky * W + ox + KW_ - 1];
      }
      float2 a = make_float2(0.0f, 0.0f);
#pragma unroll
      for (int ky = 0; ky < KH_; ++ky)
#pragma unroll
        for (int kx = 0; kx < KW_; ++kx)
          a = __ffma2_rn(make_float2(win[ky][kx], win[ky][kx]), w2[ky * KW_ + kx], a);
      *reinterpret_cast<float2*>(out + (int64_t)ox * Cout) = a;
    }
  }
}

// ---- Weight gradient, single input channel, fixed KH x KW: sliding windows
//
// dW[o, k] = sum over (m, oy, ox) of dI[m, oy, ox, o] * X[m, oy+ky, ox+kx].
// Thread t owns output row oy = t / CG and channel pair cg = t % CG (CG =
// Cout/2) and keeps both channels' KH*KW tap sums in fp32 (a float2 per
// tap).  For each of the block's images (m = b, b + G, ... in order) it
// walks its row left to right with the KH x KW input window in registers
// (KH new values a column, as in the forward) and reads one bf16 pair of
// dL/dI a pixel straight from the staged raw rows: per pixel KH + 1
// shared-memory loads for KH*KW paired FMAs.  Images are staged with
// cp.async, double-buffered; the input map is expanded to fp32.  At the end
// the Ho rows' sums are added in row order through shared memory into the
// block partial part[b][o][k], so the result is the same on every call.
constexpr int kSlideDwBlocks = 456;  // fixed block count (3 per SM of 152)

// At most 96 registers a thread (92 for 5x5: 25 float2 sums, the 5x5 window,
// no spills), so three blocks of the CSNN's first layer (24 rows x 8
// channel pairs: 192 threads) fit on an SM and the 456 blocks run in one
// wave (with 608, a third of them waited for a second wave: 12 images a
// block's slot instead of 8).

template <int KH_, int KW_>
__global__ void __maxnreg__(96) conv_slide_dw_kernel(
    const __nv_bfloat16* __restrict__ X, const __nv_bfloat16* __restrict__ dI,
    float* __restrict__ part, int64_t M, int H, int W, int Cout, int vec) {
  constexpr int KK = KH_ * KW_;
  extern __shared__ __align__(16) unsigned char dsm[];
  const int Ho = H - KH_ + 1, Wo = W - KW_ + 1, P = Ho * Wo;
  const int img = H * W, pix = P * Cout;
  const int rx = (img * 2 + 15) & ~15, rd = (pix * 2 + 15) & ~15;  // raw bytes
  auto raw = [&](int b) { return dsm + b * (rx + rd); };             // two raw buffers
  float* sx = reinterpret_cast<float*>(dsm + 2 * (rx + rd));         // [img] fp32
  const int CG = Cout / 2;
  const int t = threadIdx.x;
  const bool active = t < Ho * CG;
  const int oy = active ? t / CG : 0, cg = active ? t - (t / CG) * CG : 0;
  const int64_t G = gridDim.x;
  grid_dep_wait();
  auto stage = [&](int64_t m, int b) {
    if (vec) {
      const unsigned char* gx = reinterpret_cast<const unsigned char*>(X + m * img);
      const unsigned char* gd = reinterpret_cast<const unsigned char*>(dI + m * pix);
      for (int c = t; c < img / 8; c += blockDim.x) cp_async16(raw(b) + 16 * c, gx + 16 * c);
      for (int c = t; c < pix / 8; c += blockDim.x) cp_async16(raw(b) + rx + 16 * c, gd + 16 * c);
    } else {
      __nv_bfloat16* hx = reinterpret_cast<__nv_bfloat16*>(raw(b));
      __nv_bfloat16* hd = reinterpret_cast<__nv_bfloat16*>(raw(b) + rx);
      for (int e = t; e < img; e += blockDim.x) hx[e] = X[m * img + e];
      for (int e = t; e < pix; e += blockDim.x) hd[e] = dI[m * pix + e];
    }
    cp_async_commit();
  };
  float2 acc[KK];
#pragma unroll
  for (int k = 0; k < KK; ++k) acc[k] = make_float2(0.0f, 0.0f);
  // image i of this block is copy group i: two groups in flight before the
  // loop, one more per image
  if ((int64_t)blockIdx.x < M) stage(blockIdx.x, 0);
  else cp_async_commit();
  if ((int64_t)blockIdx.x + G < M) stage(blockIdx.x + G, 1);
  else cp_async_commit();
  int i = 0;
  for (int64_t m = blockIdx.x; m < M; m += G, ++i) {
    const int b = i & 1;
    cp_async_wait_all_but_one();  // image m's copies have landed (m + G may be in flight)
    __syncthreads();              // ... for every thread's copies
    const __nv_bfloat16* hx = reinterpret_cast<const __nv_bfloat16*>(raw(b));
    if (vec) {
      for (int v = t; v < img / 8; v += blockDim.x)
        unpack8(reinterpret_cast<const uint4*>(hx)[v], sx + 8 * v);
    } else {
      for (int e = t; e < img; e += blockDim.x) sx[e] = __bfloat162float(hx[e]);
    }
    __syncthreads();  // the fp32 map is complete
    if (active) {
      const float* row = sx + oy * W;
      const __nv_bfloat162* g2 =
          reinterpret_cast<const __nv_bfloat162*>(raw(b) + rx) + (int64_t)oy * Wo * CG + cg;
      float win[KH_][KW_];
#pragma unroll
      for (int ky = 0; ky < KH_; ++ky)
#pragma unroll
        for (int kx = 1; kx < KW_; ++kx) win[ky][kx] = row[ky * W + kx - 1];
#pragma unroll 2
      for (int ox = 0; ox < Wo; ++ox) {
#pragma unroll
        for (int ky = 0; ky < KH_; ++ky) {
#pragma unroll
          for (int kx = 0; kx < KW_ - 1; ++kx) win[ky][kx] = win[ky][kx + 1];
          win[ky][KW_ - 1] = row[ky * W + ox + KW_ - 1];
        }
        const float2 g = __bfloat1622float2(g2[ox * CG]);
#pragma unroll
        for (int ky = 0; ky < KH_; ++ky)
#pragma unroll
          for (int kx = 0; kx < KW_; ++kx)
            acc[ky * KW_ + kx] =
                __ffma2_rn(make_float2(win[ky][kx], win[ky][kx]), g, acc[ky * KW_ + kx]);
      }
    }
    __syncthreads();  // raw buffer b and the fp32 map are no longer read
    if (m + 2 * G < M) stage(m + 2 * G, b);
    else cp_async_commit();  // an empty group keeps the wait count uniform
  }
  // every copy has landed (the last groups are empty) before the staging
  // memory holds the row sums: red[(oy*CG + cg)*KK + k] = both channels
  asm volatile("cp.async.wait_all;" ::: "memory");
  __syncthreads();
  float2* red = reinterpret_cast<float2*>(dsm);
  if (active) {
#pragma unroll
    for (int k = 0; k < KK; ++k) red[(oy * CG + cg) * KK + k] = acc[k];
  }
  __syncthreads();
  for (int e = t; e < Cout * KK; e += blockDim.x) {
    const int o = e / KK, k = e - o * KK;
    const int c2 = o >> 1;
    float s = 0.0f;
    for (int r = 0; r < Ho; ++r) {
      const float2 v = red[(r * CG + c2) * KK + k];
      s += (o & 1) ? v.y : v.x;
    }
    part[((int64_t)blockIdx.x * Cout + o) * KK + k] = s;
  }
}

// dW[o, k] = sum of the G block partials, 0 for k >= K: one warp per
// output, lane l adding partials l, l + 32, ... in order, then a fixed
// shuffle tree over the lanes.
__global__ void conv_small_dw_sum(const float* __restrict__ part, float* __restrict__ dW, int G,
                                  int Cout, int K, int ldw) {
  grid_dep_wait();
  const int e = (int)((blockIdx.x * (int64_t)blockDim.x + threadIdx.x) >> 5);
  const int lane = threadIdx.x & 31;
  if (e >= Cout * ldw) return;  // warp-uniform
  const int o = e / ldw, k = e - o * ldw;
  float s = 0.0f;
  if (k < K)
    for (int b = lane; b < G; b += 32) s += part[((int64_t)b * Cout + o) * K + k];
#pragma unroll
  for (int d = 16; d > 0; d >>= 1) s += __shfl_xor_sync(0xffffffffu, s, d);
  if (lane == 0) dW[e] = s;
}

snn_status_t check_small(int64_t M, int64_t H, int64_t W, int64_t Cin, int64_t Cout, int64_t KH,
                         int64_t KW, int64_t ldw) {
  if (M < 0 || Cin < 1 || KH < 1 || KW < 1 || H < KH || W < KW) return SNN_ERR_INVALID_ARG;
  if (Cout < 1 || ldw < KH * KW * Cin) return SNN_ERR_INVALID_ARG;
  if (KH * KW * Cin > kMaxK || Cout > kMaxCout || Cout % 4 != 0 || H * W * Cin > kMaxImage)
    return SNN_ERR_UNSUPPORTED;
  if (M > INT_MAX) return SNN_ERR_INVALID_ARG;
  return SNN_OK;
}

// The sliding-window weight gradient applies: one input channel, a 5x5 or
// 3x3 filter, a thread for each (output row, channel pair) of an image in
// one block, and its staging (two raw image buffers and the fp32 map), and
// later its row sums, within shared memory.  *smem: the bytes it takes.
bool slide_dw_ok(int64_t H, int64_t W, int64_t Cin, int64_t Cout, int64_t KH, int64_t KW,
                 size_t* smem) {
  if (Cin != 1 || !((KH == 5 && KW == 5) || (KH == 3 && KW == 3))) return false;
  const int64_t Ho = H - KH + 1, Wo = W - KW + 1;
  if (Ho * (Cout / 2) > kSlideMaxThreads) return false;
  const size_t rx = ((size_t)(H * W) * 2 + 15) / 16 * 16;
  const size_t rd = ((size_t)(Ho * Wo * Cout) * 2 + 15) / 16 * 16;
  const size_t staging = 2 * (rx + rd) + (size_t)(H * W) * sizeof(float);
  const size_t sums = (size_t)(Ho * (Cout / 2) * KH * KW) * 2 * sizeof(float);
  *smem = staging > sums ? staging : sums;
  return *smem <= 200 * 1024;
}

// Blocks (= partials) of the weight gradient: a fixed count per kernel, so
// that a shape always sums in the same order.
int64_t dw_blocks(int64_t M, int64_t H, int64_t W, int64_t Cin, int64_t Cout, int64_t KH,
                  int64_t KW) {
  size_t smem = 0;
  const int64_t cap = slide_dw_ok(H, W, Cin, Cout, KH, KW, &smem) ? kSlideDwBlocks : kDwBlocks;
  return M < cap ? (M > 0 ? M : 1) : cap;
}

}  // namespace
}  // namespace snn

using namespace snn;

extern "C" snn_status_t snn_conv2d_small_fwd_nhwc(int64_t M, int64_t H, int64_t W, int64_t Cin,
                                                  int64_t Cout, int64_t KH, int64_t KW,
                                                  int64_t ldw, const void* X, const void* Wt,
                                                  float* I, snn_stream_t stream) {
  const snn_status_t s = check_small(M, H, W, Cin, Cout, KH, KW, ldw);
  if (s != SNN_OK) return s;
  if (M == 0) return SNN_OK;
  if (!X || !Wt || !I) return SNN_ERR_INVALID_ARG;
  if (reinterpret_cast<uintptr_t>(I) & 15u) return SNN_ERR_ALIGNMENT;
  if ((reinterpret_cast<uintptr_t>(X) | reinterpret_cast<uintptr_t>(Wt)) & 1u) return SNN_ERR_ALIGNMENT;
  const int Ho = (int)(H - KH + 1), Wo = (int)(W - KW + 1);
  const int units = Ho * ((Wo + 1) / 2) * (int)(Cout / 4);  // (pixel pair, channel group)
  const int passes = (units + 255) / 256;
  const int threads = ((units + passes - 1) / passes + 31) / 32 * 32;
  const int img = (int)(H * W * Cin);
  const size_t smem = (size_t)img * sizeof(float);
  const int vec = (img % 8 == 0 && (reinterpret_cast<uintptr_t>(X) & 15u) == 0 &&
                   img / 8 <= kPreVec * threads) ? 1 : 0;
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  const __nv_bfloat16* x = static_cast<const __nv_bfloat16*>(X);
  const __nv_bfloat16* w = static_cast<const __nv_bfloat16*>(Wt);
  int dev0 = 0, sms0 = 152;
  if (cudaGetDevice(&dev0) == cudaSuccess) cudaDeviceGetAttribute(&sms0, cudaDevAttrMultiProcessorCount, dev0);
  const int slide_thr = Ho * (int)(Cout / 2);
  if (Cin == 1 && ((KH == 5 && KW == 5) || (KH == 3 && KW == 3)) && slide_thr <= kSlideMaxThreads) {
    const int thr = (slide_thr + 31) / 32 * 32;
    const int vec1 = (img % 8 == 0 && (reinterpret_cast<uintptr_t>(X) & 15u) == 0 &&
                      img / 8 <= kPreVec * thr) ? 1 : 0;
    const void* ks = KH == 5 ? (const void*)conv_slide_fwd_kernel<5, 5> : (const void*)conv_slide_fwd_kernel<3, 3>;
    int per = 1;
    if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per, ks, thr, smem) != cudaSuccess || per < 1) per = 1;
    const int64_t g = M < (int64_t)sms0 * per ? M : (int64_t)sms0 * per;
    const cudaError_t e =
        KH == 5 ? launch_pdl(conv_slide_fwd_kernel<5, 5>, dim3((unsigned)g), dim3(thr), smem, st, x, w, I, M,
                             (int)H, (int)W, (int)Cout, (int)ldw, vec1)
                : launch_pdl(conv_slide_fwd_kernel<3, 3>, dim3((unsigned)g), dim3(thr), smem, st, x, w, I, M,
                             (int)H, (int)W, (int)Cout, (int)ldw, vec1);
    return e == cudaSuccess ? SNN_OK : SNN_ERR_CUDA;
  }
  const void* k = (KH == 5 && KW == 5 && Cin == 1) ? (const void*)conv_small_fwd_kernel<5, 5, 1>
                  : (KH == 3 && KW == 3 && Cin == 1) ? (const void*)conv_small_fwd_kernel<3, 3, 1>
                                                     : (const void*)conv_small_fwd_kernel<0, 0, 0>;
  // persistent blocks: as many as fit on the GPU at once (at most one per image)
  int dev = 0, sms = 152, per_sm = 1;
  if (cudaGetDevice(&dev) == cudaSuccess) cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, k, threads, smem) != cudaSuccess || per_sm < 1)
    per_sm = 1;
  const int64_t slots = (int64_t)sms * per_sm;
  const int64_t grid = M < slots ? M : slots;
  cudaError_t e;
  if (KH == 5 && KW == 5 && Cin == 1)
    e = launch_pdl(conv_small_fwd_kernel<5, 5, 1>, dim3((unsigned)grid), dim3(threads), smem, st,
                   x, w, I, M, (int)H, (int)W, (int)Cin, (int)Cout, (int)KH, (int)KW, (int)ldw, vec);
  else if (KH == 3 && KW == 3 && Cin == 1)
    e = launch_pdl(conv_small_fwd_kernel<3, 3, 1>, dim3((unsigned)grid), dim3(threads), smem, st,
                   x, w, I, M, (int)H, (int)W, (int)Cin, (int)Cout, (int)KH, (int)KW, (int)ldw, vec);
  else
    e = launch_pdl(conv_small_fwd_kernel<0, 0, 0>, dim3((unsigned)grid), dim3(threads), smem, st,
                   x, w, I, M, (int)H, (int)W, (int)Cin, (int)Cout, (int)KH, (int)KW, (int)ldw, vec);
  return e == cudaSuccess ? SNN_OK : SNN_ERR_CUDA;
}

extern "C" size_t snn_conv2d_small_dw_workspace_bytes(int64_t M, int64_t H, int64_t W,
                                                      int64_t Cin, int64_t Cout, int64_t KH,
                                                      int64_t KW) {
  if (check_small(M, H, W, Cin, Cout, KH, KW, KH * KW * Cin) != SNN_OK) return 0;
  return (size_t)dw_blocks(M, H, W, Cin, Cout, KH, KW) * Cout * KH * KW * Cin * sizeof(float);
}

extern "C" snn_status_t snn_conv2d_small_dw_nhwc(int64_t M, int64_t H, int64_t W, int64_t Cin,
                                                 int64_t Cout, int64_t KH, int64_t KW, int64_t ldw,
                                                 const void* X, const void* dI, float* dW,
                                                 void* ws, size_t ws_bytes, snn_stream_t stream) {
  const snn_status_t s = check_small(M, H, W, Cin, Cout, KH, KW, ldw);
  if (s != SNN_OK) return s;
  if (!dW) return SNN_ERR_INVALID_ARG;
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  if (M == 0)
    return cudaMemsetAsync(dW, 0, (size_t)Cout * ldw * sizeof(float), st) == cudaSuccess ? SNN_OK
                                                                                         : SNN_ERR_CUDA;
  if (!X || !dI) return SNN_ERR_INVALID_ARG;
  if (!ws || ws_bytes < snn_conv2d_small_dw_workspace_bytes(M, H, W, Cin, Cout, KH, KW))
    return SNN_ERR_WORKSPACE;
  if ((reinterpret_cast<uintptr_t>(ws) | reinterpret_cast<uintptr_t>(dW)) & 15u)
    return SNN_ERR_ALIGNMENT;
  if ((reinterpret_cast<uintptr_t>(X) | reinterpret_cast<uintptr_t>(dI)) & 1u) return SNN_ERR_ALIGNMENT;
  const int K = (int)(KH * KW * Cin);
  const int64_t G = dw_blocks(M, H, W, Cin, Cout, KH, KW);
  float* part = static_cast<float*>(ws);
  cudaError_t e = cudaSuccess;
  size_t slide_smem = 0;
  if (slide_dw_ok(H, W, Cin, Cout, KH, KW, &slide_smem)) {
    const int thr = ((int)((H - KH + 1) * (Cout / 2)) + 31) / 32 * 32;
    // raw 16-byte copies of whole images: both image sizes a multiple of 8
    // elements, both bases 16-byte aligned (dI stays bf16 in shared memory)
    const int vec1 = ((H * W) % 8 == 0 && ((H - KH + 1) * (W - KW + 1) * Cout) % 8 == 0 &&
                      ((reinterpret_cast<uintptr_t>(X) | reinterpret_cast<uintptr_t>(dI)) & 15u) == 0)
                         ? 1 : 0;
    const void* ks = KH == 5 ? (const void*)conv_slide_dw_kernel<5, 5> : (const void*)conv_slide_dw_kernel<3, 3>;
    if (slide_smem > 48 * 1024 &&
        cudaFuncSetAttribute(ks, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)slide_smem) != cudaSuccess)
      return SNN_ERR_CUDA;
    const __nv_bfloat16* x1 = static_cast<const __nv_bfloat16*>(X);
    const __nv_bfloat16* d1 = static_cast<const __nv_bfloat16*>(dI);
    e = KH == 5 ? launch_pdl(conv_slide_dw_kernel<5, 5>, dim3((unsigned)G), dim3(thr), slide_smem, st, x1,
                             d1, part, M, (int)H, (int)W, (int)Cout, vec1)
                : launch_pdl(conv_slide_dw_kernel<3, 3>, dim3((unsigned)G), dim3(thr), slide_smem, st, x1,
                             d1, part, M, (int)H, (int)W, (int)Cout, vec1);
    if (e != cudaSuccess) return SNN_ERR_CUDA;
    const int n = (int)(Cout * ldw);  // one warp each
    e = launch_pdl(conv_small_dw_sum, dim3((unsigned)((n + 7) / 8)), dim3(256), 0, st,
                   static_cast<const float*>(part), dW, (int)G, (int)Cout, K, (int)ldw);
    return e == cudaSuccess ? SNN_OK : SNN_ERR_CUDA;
  }
  const int P = (int)((H - KH + 1) * (W - KW + 1));
  const int img = (int)(H * W * Cin);
  const int64_t pix = (int64_t)P * Cout;
  const size_t rawb = 2 * (((size_t)img * 2 + 15) / 16 * 16 + ((size_t)pix * 2 + 15) / 16 * 16);
  const size_t smem = rawb + (size_t)(((img + 3) & ~3) + pix) * sizeof(float);
  if (smem > 200 * 1024) return SNN_ERR_UNSUPPORTED;
  const int vec = (img % 8 == 0 && Cout % 8 == 0 &&
                   ((reinterpret_cast<uintptr_t>(X) | reinterpret_cast<uintptr_t>(dI)) & 15u) == 0)
                      ? 1 : 0;
  const __nv_bfloat16* x = static_cast<const __nv_bfloat16*>(X);
  const __nv_bfloat16* d = static_cast<const __nv_bfloat16*>(dI);
  const void* k = (KH == 5 && KW == 5 && Cin == 1) ? (const void*)conv_small_dw_kernel<5, 5, 1, 25>
                  : (K <= 16) ? (const void*)conv_small_dw_kernel<0, 0, 0, 16>
                              : (const void*)conv_small_dw_kernel<0, 0, 0, 32>;
  e = smem > 48 * 1024 ? cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem)
                       : cudaSuccess;
  if (e != cudaSuccess) return SNN_ERR_CUDA;
  if (KH == 5 && KW == 5 && Cin == 1)
    e = launch_pdl(conv_small_dw_kernel<5, 5, 1, 25>, dim3((unsigned)G), dim3(kDwThreads), smem, st,
                   x, d, part, M, (int)H, (int)W, (int)Cin, (int)Cout, (int)KH, (int)KW, vec);
  else if (K <= 16)
    e = launch_pdl(conv_small_dw_kernel<0, 0, 0, 16>, dim3((unsigned)G), dim3(kDwThreads), smem, st,
                   x, d, part, M, (int)H, (int)W, (int)Cin, (int)Cout, (int)KH, (int)KW, vec);
  else
    e = launch_pdl(conv_small_dw_kernel<0, 0, 0, 32>, dim3((unsigned)G), dim3(kDwThreads), smem, st,
                   x, d, part, M, (int)H, (int)W, (int)Cin, (int)Cout, (int)KH, (int)KW, vec);
  if (e != cudaSuccess) return SNN_ERR_CUDA;
  const int n = (int)(Cout * ldw);  // one warp each
  e = launch_pdl(conv_small_dw_sum, dim3((unsigned)((n + 7) / 8)), dim3(256), 0, st,
                 static_cast<const float*>(part), dW, (int)G, (int)Cout, K, (int)ldw);
  return e == cudaSuccess ? SNN_OK : SNN_ERR_CUDA;
}
