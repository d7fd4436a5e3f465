// Deterministic reduction of per-lane parameter-gradient partials (fp32, one
// per lane, already summed over t by the scan) into the parameter's shape:
// scalar, per neuron [N] (sum over b) or per channel [C] (sum over b and the
// channel's H*W positions).  Cross-lane sums run in fp64 in a fixed order, so
// repeated calls give identical bits.
#include "scan_host.cuh"

namespace snn {

namespace {

constexpr int kRedThreads = 256;

__device__ __forceinline__ double block_sum(double v, double* sh) {
  sh[threadIdx.x] = v;
  __syncthreads();
  for (int s = blockDim.x / 2; s > 0; s >>= 1) {
    if ((int)threadIdx.x < s) sh[threadIdx.x] += sh[threadIdx.x + s];
    __syncthreads();
  }
  return sh[0];
}

// Stage 1 of the scalar sum: block b sums lanes [b*chunk, (b+1)*chunk).
__global__ void __launch_bounds__(kRedThreads) reduce_scalar_blocks(const float* part, int64_t L,
                                                                     int64_t chunk, double* out) {
  __shared__ double sh[kRedThreads];
  const int64_t lo = (int64_t)blockIdx.x * chunk;
  const int64_t hi = min(L, lo + chunk);
  double acc = 0.0;
  for (int64_t l = lo + threadIdx.x; l < hi; l += blockDim.x) acc += (double)part[l];
  const double s = block_sum(acc, sh);
  if (threadIdx.x == 0) out[blockIdx.x] = s;
}

__global__ void __launch_bounds__(kRedThreads) reduce_scalar_final(const double* in, int n,
                                                                    float* out) {
  __shared__ double sh[kRedThreads];
  double acc = 0.0;
  for (int i = threadIdx.x; i < n; i += blockDim.x) acc += in[i];
  const double s = block_sum(acc, sh);
  if (threadIdx.x == 0) out[0] = (float)s;
}

// One thread per neuron n: sum over b of part[b*N + n].
__global__ void __launch_bounds__(kRedThreads) reduce_per_neuron(const float* part, int64_t B,
                                                                  int64_t N, float* out) {
  const int64_t n = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (n >= N) return;
  double acc = 0.0;
  for (int64_t b = 0; b < B; ++b) acc += (double)part[b * N + n];
  out[n] = (float)acc;
}

// One block per channel c: neurons n = (r*C + c)*HW + h for r < N/(C*HW).
__global__ void __launch_bounds__(kRedThreads) reduce_per_channel(const float* part, int64_t B,
                                                                   int64_t N, int64_t C,
                                                                   int64_t HW, float* out) {
  __shared__ double sh[kRedThreads];
  const int64_t c = blockIdx.x;
  const int64_t R = N / (C * HW);
  const int64_t per_b = R * HW;
  const int64_t total = B * per_b;
  double acc = 0.0;
  for (int64_t k = threadIdx.x; k < total; k += blockDim.x) {
    const int64_t b = k / per_b, rem = k % per_b;
    const int64_t r = rem / HW, h = rem % HW;
    acc += (double)part[b * N + (r * C + c) * HW + h];
  }
  const double s = block_sum(acc, sh);
  if (threadIdx.x == 0) out[c] = (float)s;
}

}  // namespace

cudaError_t launch_param_reduce(const float* part, int64_t B, int64_t N, int64_t C, int64_t HW,
                                int mode, double* scratch, int scratch_len, float* out,
                                cudaStream_t stream) {
  const int64_t L = B * N;
  if (mode == PM_SCALAR) {
    const int64_t chunk_min = 4096;
    int64_t nb = ceil_div(L, chunk_min);
    if (nb > scratch_len) nb = scratch_len;
    if (nb < 1) nb = 1;
    const int64_t chunk = ceil_div(L > 0 ? L : 1, nb);
    nb = ceil_div(L > 0 ? L : 1, chunk);
    reduce_scalar_blocks<<<(unsigned)nb, kRedThreads, 0, stream>>>(part, L, chunk, scratch);
    reduce_scalar_final<<<1, kRedThreads, 0, stream>>>(scratch, (int)nb, out);
  } else if (mode == PM_PER_NEURON) {
    if (N > 0) reduce_per_neuron<<<(unsigned)ceil_div(N, kRedThreads), kRedThreads, 0, stream>>>(part, B, N, out);
  } else {
    if (C > 0) reduce_per_channel<<<(unsigned)C, kRedThreads, 0, stream>>>(part, B, N, C, HW, out);
  }
  return cudaGetLastError();
}

}  // namespace snn
