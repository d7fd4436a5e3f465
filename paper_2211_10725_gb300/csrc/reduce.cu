// Deterministic reduction of per-lane parameter-gradient partials (fp32, one
// per lane, already summed over t by the scan) into the parameter's shape:
// scalar, per neuron [N] (sum over b) or per channel [C] (sum over b and the
// channel's H*W positions).  Each thread adds its own run of lanes in fp32
// (tens of terms: an error of a few 1e-6 of their magnitudes), and
// everything above that in compensated fp32: a running sum and the rounding
// error of its additions (Knuth's two-sum), close to fp64's accuracy for
// these sums without fp64 arithmetic, which is slow on this part (with one
// fp64 add per lane the per-neuron reduction of the 524,288-lane workload
// took 11.5 us).  Every sum is taken in a fixed order, so repeated calls
// give identical bits.
//
// One launch reduces every parameter that shares a layout (blockIdx.z picks
// the parameter).  Scalar and per-channel: block (x, y) of a parameter sums
// split y of output group x into scratch (one (sum, error) pair in each
// 8-byte slot); the last of a group's splits to finish (a ticket taken
// after its partial is published) adds the group's partials in split order
// and writes the result, then resets the group's ticket to zero for the
// next call.  Per neuron, a neuron's B partials fit one block, which sums
// them in a single pass.
#include "scan_host.cuh"

namespace snn {

namespace {

constexpr int kRedThreads = 256;
constexpr int64_t kChanChunk = 8192;  // lanes per block of the channel-last reduction (32 per thread)
constexpr int64_t kNeuronSplit = 8;

// (sum, error) += x: the rounding error of the addition kept in .y
// (two-sum; every operation rounded to nearest, none fused).
__device__ __forceinline__ float2 two_add(float2 a, float x) {
  const float s = __fadd_rn(a.x, x);
  const float z = __fadd_rn(s, -a.x);
  const float e = __fadd_rn(__fadd_rn(a.x, -__fadd_rn(s, -z)), __fadd_rn(x, -z));
  return make_float2(s, __fadd_rn(a.y, e));
}
// (sum, error) += (sum', error')
__device__ __forceinline__ float2 pair_add(float2 a, float2 b) {
  a = two_add(a, b.x);
  a.y = __fadd_rn(a.y, b.y);
  return a;
}
// The pair's value; a non-finite sum is returned as it is (its error term
// is NaN once an infinity entered the sum).
__device__ __forceinline__ float pair_value(float2 a) {
  return isfinite(a.x) ? __fadd_rn(a.x, a.y) : a.x;
}

// The block's values added in a fixed tree.
__device__ __forceinline__ float2 block_sum(float2 v, float2* sh) {
  sh[threadIdx.x] = v;
  __syncthreads();
  for (int s = blockDim.x / 2; s > 0; s >>= 1) {
    if ((int)threadIdx.x < s) sh[threadIdx.x] = pair_add(sh[threadIdx.x], sh[threadIdx.x + s]);
    __syncthreads();
  }
  const float2 r = sh[0];
  __syncthreads();
  return r;
}

struct ReduceJob {
  const float* part;  // per-lane partials [B*N]
  float* out;         // reduced gradient
  float2* scratch;    // block partials, (sum, error) pairs
  int* tickets;       // one per output group, zero between calls
};

struct ReduceJobs {
  ReduceJob job[3];
};

// True in every thread of the block that finished a group last.
__device__ __forceinline__ bool last_of_group(int* ticket, int splits) {
  __shared__ int last;
  __threadfence();  // this block's partial is visible before its ticket
  __syncthreads();
  if (threadIdx.x == 0) last = atomicAdd(ticket, 1) == splits - 1;
  __syncthreads();
  if (last) __threadfence();  // and the other blocks' partials before the sum
  return last;
}

// Scalar: group 0, split y sums lanes [y*chunk, (y+1)*chunk).
__global__ void __launch_bounds__(kRedThreads) reduce_scalar(ReduceJobs js, int64_t L,
                                                              int64_t chunk) {
  __shared__ float2 sh[kRedThreads];
  grid_dep_wait();
  const ReduceJob& j = js.job[blockIdx.z];
  const int S = gridDim.y;
  const int64_t lo = (int64_t)blockIdx.y * chunk;
  const int64_t hi = min(L, lo + chunk);
  // a thread's run of lanes (16 at the default chunk) in fp32, in order;
  // everything above compensated
  float acc = 0.0f;
  for (int64_t l = lo + threadIdx.x; l < hi; l += blockDim.x) acc += j.part[l];
  const float2 s = block_sum(make_float2(acc, 0.0f), sh);
  if (threadIdx.x == 0) j.scratch[blockIdx.y] = s;
  if (!last_of_group(&j.tickets[0], S)) return;
  float2 t = make_float2(0.0f, 0.0f);
  for (int i = threadIdx.x; i < S; i += blockDim.x) t = pair_add(t, j.scratch[i]);
  const float2 total = block_sum(t, sh);
  if (threadIdx.x == 0) {
    j.out[0] = pair_value(total);
    j.tickets[0] = 0;
  }
}

// Per neuron, in one pass: block x covers neurons [32x, 32x + 32), warp y
// sums split y of the samples, [B*y/S, B*(y+1)/S), in fp32 in order; warp 0
// then adds the S split sums of each neuron, compensated, in split order.
// The whole sum over b of a neuron lives in one block, so no partial leaves
// it and no ticket or second round trip through memory is needed.
__global__ void __launch_bounds__(kRedThreads) reduce_per_neuron(ReduceJobs js, int64_t B,
                                                                  int64_t N) {
  __shared__ float sh[kNeuronSplit][32];
  grid_dep_wait();
  const ReduceJob& j = js.job[blockIdx.z];
  const int lid = threadIdx.x & 31, s = threadIdx.x >> 5;
  const int S = blockDim.x >> 5;
  const int64_t n = (int64_t)blockIdx.x * 32 + lid;
  if (n < N) {
    // the split's samples (8 at B = 64) in fp32, in order; the splits compensated
    const int64_t b0 = B * s / S, b1 = B * (s + 1) / S;
    float acc = 0.0f;
    for (int64_t b = b0; b < b1; ++b) acc += j.part[b * N + n];
    sh[s][lid] = acc;
  }
  __syncthreads();
  if (s == 0 && n < N) {
    float2 acc = make_float2(0.0f, 0.0f);
    for (int q = 0; q < S; ++q) acc = two_add(acc, sh[q][lid]);
    j.out[n] = pair_value(acc);
  }
}

// Per channel: group x = channel c, split y sums the runs j = y, y + S, ...
// of channel c, where run j = (b, r) is the HW contiguous lanes of neurons
// (r*C + c)*HW .. +HW of sample b (r < N/(C*HW)).  The block's runs are
// flattened so that short runs still keep every thread busy.
__global__ void __launch_bounds__(kRedThreads) reduce_per_channel(ReduceJobs js, int64_t B,
                                                                   int64_t N, int64_t C,
                                                                   int64_t HW) {
  __shared__ float2 sh[kRedThreads];
  grid_dep_wait();
  const ReduceJob& j = js.job[blockIdx.z];
  const int64_t c = blockIdx.x, s = blockIdx.y, S = gridDim.y;
  const int64_t R = N / (C * HW);
  const int64_t runs = (B * R - s + S - 1) / S;  // runs j = s + q*S, q < runs
  float acc = 0.0f;  // a thread's elements in fp32, in order; the block's compensated
  for (int64_t e = threadIdx.x; e < runs * HW; e += blockDim.x) {
    const int64_t q = e / HW, h = e - q * HW;
    const int64_t jr = s + q * S;
    const int64_t b = jr / R, r = jr - b * R;
    acc += j.part[b * N + (r * C + c) * HW + h];
  }
  const float2 v = block_sum(make_float2(acc, 0.0f), sh);
  if (threadIdx.x == 0) j.scratch[c * S + s] = v;
  if (!last_of_group(&j.tickets[c], (int)S)) return;
  if (threadIdx.x < 32) {  // lane l adds splits l, l + 32, ... in order, then a fixed tree
    float2 t = make_float2(0.0f, 0.0f);
    for (int64_t q = threadIdx.x; q < S; q += 32) t = pair_add(t, j.scratch[c * S + q]);
#pragma unroll
    for (int d = 16; d > 0; d >>= 1) {
      const float2 o = make_float2(__shfl_xor_sync(0xffffffffu, t.x, d),
                                   __shfl_xor_sync(0xffffffffu, t.y, d));
      t = pair_add(t, o);
    }
    if (threadIdx.x == 0) {
      j.out[c] = pair_value(t);
      j.tickets[c] = 0;
    }
  }
}

// Per channel with one position per channel run (HW = 1: channel-last
// lanes, the channel of lane l is l % C) and C dividing the block size:
// block x sums lanes [x*chunk, (x+1)*chunk), chunk a multiple of the block
// size, so thread t only meets channel t % C and its loads are coalesced.
// The threads of a channel are added in thread order; the last block adds
// the block partials of each channel in a fixed two-level order spread over
// all its threads.
__global__ void __launch_bounds__(kRedThreads) reduce_channel_last(ReduceJobs js, int64_t L,
                                                                    int64_t chunk, int C) {
  __shared__ float2 sh[kRedThreads];
  grid_dep_wait();
  const ReduceJob& j = js.job[blockIdx.z];
  const int64_t lo = (int64_t)blockIdx.x * chunk;
  const int64_t hi = min(L, lo + chunk);
  // a thread's run of lanes (32 at kChanChunk) in fp32, everything above
  // compensated
  float acc = 0.0f;
#pragma unroll 8
  for (int64_t l = lo + threadIdx.x; l < hi; l += kRedThreads) acc += j.part[l];
  sh[threadIdx.x] = make_float2(acc, 0.0f);
  __syncthreads();
  if ((int)threadIdx.x < C) {
    float2 t = make_float2(0.0f, 0.0f);
    for (int q = threadIdx.x; q < kRedThreads; q += C) t = pair_add(t, sh[q]);
    j.scratch[(int64_t)blockIdx.x * C + threadIdx.x] = t;
  }
  if (!last_of_group(&j.tickets[0], (int)gridDim.x)) return;
  // thread (c, p) = (t % C, t / C) adds the block partials p, p + P, ... of
  // channel c in order (P = 256 / C parts, independent loads in flight);
  // then thread c adds its channel's P parts in order
  const int P = kRedThreads / C;
  const int c = threadIdx.x % C, pp = threadIdx.x / C;
  float2 t = make_float2(0.0f, 0.0f);
#pragma unroll 8
  for (int q = pp; q < (int)gridDim.x; q += P) t = pair_add(t, j.scratch[(int64_t)q * C + c]);
  __syncthreads();  // every thread is done with sh
  sh[threadIdx.x] = t;
  __syncthreads();
  if ((int)threadIdx.x < C) {
    float2 total = make_float2(0.0f, 0.0f);
    for (int k = 0; k < P; ++k) total = pair_add(total, sh[k * C + threadIdx.x]);
    j.out[threadIdx.x] = pair_value(total);
  }
  if (threadIdx.x == 0) j.tickets[0] = 0;
}

}  // namespace

cudaError_t launch_param_reduce(const ParamReduce* p, int n, int64_t B, int64_t N, int64_t C,
                                int64_t HW, int mode, int64_t scratch_len, cudaStream_t stream) {
  if (n <= 0) return cudaSuccess;
  if (n > 3) return cudaErrorInvalidValue;
  ReduceJobs js;
  // the scratch's 8-byte slots hold (sum, error) pairs
  for (int k = 0; k < n; ++k)
    js.job[k] = ReduceJob{p[k].part, p[k].out, reinterpret_cast<float2*>(p[k].scratch), p[k].tickets};
  const int64_t L = B * N;
  if (mode == PM_SCALAR) {
    const int64_t chunk_min = 4096;
    int64_t nb = ceil_div(L, chunk_min);
    if (nb > scratch_len) nb = scratch_len;
    if (nb > 65535) nb = 65535;
    if (nb < 1) nb = 1;
    const int64_t chunk = ceil_div(L > 0 ? L : 1, nb);
    nb = ceil_div(L > 0 ? L : 1, chunk);
    const cudaError_t e = launch_pdl(reduce_scalar, dim3(1, (unsigned)nb, (unsigned)n),
                                     dim3(kRedThreads), 0, stream, js, L, chunk);
    if (e != cudaSuccess) return e;
  } else if (mode == PM_PER_NEURON) {
    if (N > 0) {
      const int64_t S = B < kNeuronSplit ? (B < 1 ? 1 : B) : kNeuronSplit;
      const cudaError_t e =
          launch_pdl(reduce_per_neuron, dim3((unsigned)ceil_div(N, 32), 1, (unsigned)n),
                     dim3((unsigned)(32 * S)), 0, stream, js, B, N);
      if (e != cudaSuccess) return e;
    }
  } else if (C > 0 && HW == 1 && kRedThreads % C == 0) {
    int64_t nb = ceil_div(L, kChanChunk);
    if (nb > scratch_len / C) nb = scratch_len / C;
    if (nb > 65535) nb = 65535;
    if (nb < 1) return cudaErrorInvalidValue;  // the workspace is sized for one block
    // kChanChunk lanes per block unless the workspace holds fewer block partials
    const int64_t chunk = ceil_div(ceil_div(L > 0 ? L : 1, nb), kRedThreads) * kRedThreads;
    nb = ceil_div(L > 0 ? L : 1, chunk);
    const cudaError_t e = launch_pdl(reduce_channel_last, dim3((unsigned)nb, 1, (unsigned)n),
                                     dim3(kRedThreads), 0, stream, js, L, chunk, (int)C);
    if (e != cudaSuccess) return e;
  } else if (C > 0) {
    const int64_t R = N / (C * HW);
    // about four blocks per SM in total, at least ~1k elements per block
    int64_t S = ceil_div(608, C);
    const int64_t by_size = ceil_div(B * R * HW, 1024);
    if (S > by_size) S = by_size;
    if (S > B * R) S = B * R;
    if (S > scratch_len / C) S = scratch_len / C;
    if (S < 1) return cudaErrorInvalidValue;  // the workspace is sized for S >= 1
    const cudaError_t e = launch_pdl(reduce_per_channel, dim3((unsigned)C, (unsigned)S, (unsigned)n),
                                     dim3(kRedThreads), 0, stream, js, B, N, C, HW);
    if (e != cudaSuccess) return e;
  }
  return cudaGetLastError();
}

}  // namespace snn
