// Deterministic reduction of per-lane parameter-gradient partials (fp32, one
// per lane, already summed over t by the scan) into the parameter's shape:
// scalar, per neuron [N] (sum over b) or per channel [C] (sum over b and the
// channel's H*W positions).  Cross-lane sums run in fp64 in a fixed order, so
// repeated calls give identical bits.
#include "scan_host.cuh"

namespace snn {

namespace {

constexpr int kRedThreads = 256;
constexpr int64_t kNeuronSplit = 8;

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

// Per-neuron sum, stage 1: block (x, s) sums samples b in [b0, b1) of
// split s for 256 neurons; stage 2 adds the splits of each neuron in order.
__global__ void __launch_bounds__(kRedThreads) reduce_per_neuron_blocks(const float* part,
                                                                         int64_t B, int64_t N,
                                                                         double* out) {
  const int64_t n = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (n >= N) return;
  const int64_t S = gridDim.y, s = blockIdx.y;
  const int64_t b0 = B * s / S, b1 = B * (s + 1) / S;
  double acc = 0.0;
  for (int64_t b = b0; b < b1; ++b) acc += (double)part[b * N + n];
  out[s * N + n] = acc;
}

__global__ void __launch_bounds__(kRedThreads) reduce_per_neuron_final(const double* in, int64_t N,
                                                                        int S, float* out) {
  const int64_t n = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (n >= N) return;
  double acc = 0.0;
  for (int s = 0; s < S; ++s) acc += in[s * N + n];
  out[n] = (float)acc;
}

// Per-channel sum, stage 1: block (c, s) sums the runs j = s, s + S, ... of
// channel c, where run j = (b, r) is the HW contiguous lanes of neurons
// (r*C + c)*HW .. +HW of sample b (r < N/(C*HW)).  The block's runs are
// flattened so that short runs still keep every thread busy.
__global__ void __launch_bounds__(kRedThreads) reduce_per_channel_blocks(
    const float* part, int64_t B, int64_t N, int64_t C, int64_t HW, double* out) {
  __shared__ double sh[kRedThreads];
  const int64_t c = blockIdx.x, s = blockIdx.y, S = gridDim.y;
  const int64_t R = N / (C * HW);
  const int64_t runs = (B * R - s + S - 1) / S;  // runs j = s + q*S, q < runs
  double acc = 0.0;
  for (int64_t e = threadIdx.x; e < runs * HW; e += blockDim.x) {
    const int64_t q = e / HW, h = e - q * HW;
    const int64_t j = s + q * S;
    const int64_t b = j / R, r = j - b * R;
    acc += (double)part[b * N + (r * C + c) * HW + h];
  }
  const double v = block_sum(acc, sh);
  if (threadIdx.x == 0) out[c * S + s] = v;
}

// Stage 2: channel c adds its S partials in order.
__global__ void __launch_bounds__(kRedThreads) reduce_per_channel_final(const double* in, int64_t C,
                                                                         int S, float* out) {
  const int64_t c = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (c >= C) return;
  double acc = 0.0;
  for (int s = 0; s < S; ++s) acc += in[c * S + s];
  out[c] = (float)acc;
}

}  // namespace

cudaError_t launch_param_reduce(const float* part, int64_t B, int64_t N, int64_t C, int64_t HW,
                                int mode, double* scratch, int64_t scratch_len, float* out,
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
    if (N > 0) {
      int64_t S = B < kNeuronSplit ? B : kNeuronSplit;
      if (S * N > scratch_len) S = scratch_len / N;
      if (S < 1) return cudaErrorInvalidValue;  // the workspace is sized for S >= 1
      reduce_per_neuron_blocks<<<dim3((unsigned)ceil_div(N, kRedThreads), (unsigned)S), kRedThreads,
                                 0, stream>>>(part, B, N, scratch);
      reduce_per_neuron_final<<<(unsigned)ceil_div(N, kRedThreads), kRedThreads, 0, stream>>>(
          scratch, N, (int)S, out);
    }
  } else if (C > 0) {
    const int64_t R = N / (C * HW);
    // about four blocks per SM in total, at least ~1k elements per block
    int64_t S = ceil_div(608, C);
    const int64_t by_size = ceil_div(B * R * HW, 1024);
    if (S > by_size) S = by_size;
    if (S > B * R) S = B * R;
    if (S > scratch_len / C) S = scratch_len / C;
    if (S < 1) return cudaErrorInvalidValue;  // the workspace is sized for S >= 1
    reduce_per_channel_blocks<<<dim3((unsigned)C, (unsigned)S), kRedThreads, 0, stream>>>(
        part, B, N, C, HW, scratch);
    reduce_per_channel_final<<<(unsigned)ceil_div(C, kRedThreads), kRedThreads, 0, stream>>>(
        scratch, C, (int)S, out);
  }
  return cudaGetLastError();
}

}  // namespace snn
