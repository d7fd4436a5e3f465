// C ABI of libsnn (declared in include/snn.h): argument checks, workspace
// layout, kernel selection.  Every check runs before anything is launched.
#include <cmath>
#include <cstring>

#include "scan_host.cuh"
#include "snn.h"

namespace snn {
namespace {

constexpr size_t kStatusBytes = 256;
constexpr uint64_t kDefaultWaitNs = 2000000000ull;

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

size_t dtype_size(int dt) { return dt == SNN_F32 ? 4 : 2; }

bool valid_dtype(int dt) { return dt == SNN_F32 || dt == SNN_BF16 || dt == SNN_F16; }

bool supported_pair(int in_dt, int io_dt) {
  return in_dt == io_dt || (in_dt == SNN_F32 && io_dt != SNN_F32);
}

int64_t param_len(int mode, const snn_scan_desc* d) {
  return mode == SNN_P_SCALAR ? 1 : (mode == SNN_P_PER_NEURON ? d->N : d->C);
}

snn_status_t check_desc(const snn_scan_desc* d) {
  if (!d) return SNN_ERR_INVALID_ARG;
  if (d->T < 0 || d->B < 0 || d->N < 0) return SNN_ERR_INVALID_ARG;
  if (d->T >= ((int64_t)1 << 31)) return SNN_ERR_INVALID_ARG;
  if (d->B > 0 && d->N > INT64_MAX / d->B) return SNN_ERR_INVALID_ARG;
  const int64_t L = d->B * d->N;
  if (d->T > 0 && L > INT64_MAX / 8 / d->T) return SNN_ERR_INVALID_ARG;
  if (!valid_dtype(d->in_dtype) || !valid_dtype(d->io_dtype)) return SNN_ERR_INVALID_ARG;
  if (d->reset < SNN_RESET_SUBTRACT || d->reset > SNN_RESET_NONE) return SNN_ERR_INVALID_ARG;
  if (d->detach_reset != 0 && d->detach_reset != 1) return SNN_ERR_INVALID_ARG;
  if (d->surrogate != SNN_SG_FAST_SIGMOID && d->surrogate != SNN_SG_ATAN) return SNN_ERR_INVALID_ARG;
  if (!(d->sg_param > 0.0f) || !std::isfinite(d->sg_param)) return SNN_ERR_INVALID_ARG;
  const int modes[3] = {d->beta_mode, d->thr_mode, d->alpha_mode};
  bool per_channel = false;
  for (int m : modes) {
    if (m < SNN_P_SCALAR || m > SNN_P_PER_CHANNEL) return SNN_ERR_INVALID_ARG;
    per_channel |= (m == SNN_P_PER_CHANNEL);
  }
  if (per_channel) {
    if (d->C < 1 || d->HW < 1) return SNN_ERR_INVALID_ARG;
    if (d->N % (d->C * d->HW) != 0) return SNN_ERR_INVALID_ARG;
  }
  if (d->save != SNN_SAVE_MEM && d->save != SNN_SAVE_RECOMPUTE) return SNN_ERR_INVALID_ARG;
  if (d->save == SNN_SAVE_RECOMPUTE && (d->ckpt_every < 1 || d->ckpt_every > 64))
    return d->ckpt_every < 1 ? SNN_ERR_INVALID_ARG : SNN_ERR_UNSUPPORTED;
  if (d->reserved0 != 0 || d->reserved1 != 0) return SNN_ERR_INVALID_ARG;
  if (d->wait_limit_ns < 0) return SNN_ERR_INVALID_ARG;
  if (!supported_pair(d->in_dtype, d->io_dtype)) return SNN_ERR_UNSUPPORTED;
  return SNN_OK;
}

size_t lane_bytes(const snn_scan_desc* d) {
  return (size_t)round_up((int64_t)d->B * d->N * 4, 256);
}

// fp64 partials of one parameter's cross-lane reduction
int64_t red_scratch(const snn_scan_desc* d) { return param_reduce_scratch(d->N, d->C); }

size_t ticket_bytes(const snn_scan_desc* d) {
  return (size_t)round_up(param_reduce_groups(d->N, d->C) * (int64_t)sizeof(int), 256);
}

size_t workspace_bytes(const snn_scan_desc* d) {
  return kStatusBytes + 3 * lane_bytes(d) + 3 * (size_t)red_scratch(d) * sizeof(double) +
         3 * ticket_bytes(d);
}

struct WsView {
  int* status;
  float* part[3];  // beta, thr, alpha (or v)
  double* scratch[3];
  int* tickets[3];
};

WsView ws_view(void* ws, const snn_scan_desc* d) {
  unsigned char* p = static_cast<unsigned char*>(ws);
  WsView v;
  v.status = reinterpret_cast<int*>(p);
  const size_t lb = lane_bytes(d);
  for (int k = 0; k < 3; ++k) v.part[k] = reinterpret_cast<float*>(p + kStatusBytes + k * lb);
  for (int k = 0; k < 3; ++k)
    v.scratch[k] = reinterpret_cast<double*>(p + kStatusBytes + 3 * lb + k * red_scratch(d) * sizeof(double));
  unsigned char* t = p + kStatusBytes + 3 * lb + 3 * red_scratch(d) * sizeof(double);
  for (int k = 0; k < 3; ++k) v.tickets[k] = reinterpret_cast<int*>(t + k * ticket_bytes(d));
  return v;
}

snn_status_t check_ptrs(std::initializer_list<const void*> ptrs) {
  for (const void* p : ptrs)
    if (p && !aligned16(p)) return SNN_ERR_ALIGNMENT;
  return SNN_OK;
}

snn_status_t check_ws(const snn_scan_desc* d, const void* ws, size_t ws_bytes) {
  if (!ws || ws_bytes < workspace_bytes(d)) return SNN_ERR_WORKSPACE;
  return aligned16(ws) ? SNN_OK : SNN_ERR_ALIGNMENT;
}

// Rows of every streamed tensor must be 16-byte multiples for the TMA path,
// and lanes come in groups of VEC per thread.
// Bytes per time step of the spike-bit rows (store mode, half io): one bit
// per lane, rows padded to 16 bytes.
int64_t spike_bits_row(const snn_scan_desc* d) { return round_up(ceil_div(d->B * d->N, 8), 16); }

bool staged_ok(const snn_scan_desc* d) {
  if (d->debug_flags & 2u) return false;  // SNN_DEBUG_FORCE_PLAIN
  const int64_t L = d->B * d->N;
  return L > 0 && L % VEC == 0 && (L * (int64_t)dtype_size(d->in_dtype)) % 16 == 0 &&
         (L * (int64_t)dtype_size(d->io_dtype)) % 16 == 0 && (L * 4) % 16 == 0;
}

ScanArgs base_args(const snn_scan_desc* d, void* ws) {
  ScanArgs a;
  std::memset(&a, 0, sizeof(a));
  a.T = d->T;
  a.L = d->B * d->N;
  a.N = d->N > 0 ? d->N : 1;
  a.C = d->C > 0 ? d->C : 1;
  a.HW = d->HW > 0 ? d->HW : 1;
  if (d->save == SNN_SAVE_RECOMPUTE) {
    a.K = d->ckpt_every;
    a.nseg = (int)ceil_div(d->T, d->ckpt_every);
  } else {
    a.K = d->T > 0 ? (int)d->T : 1;
    a.nseg = d->T > 0 ? 1 : 0;
  }
  a.reset = d->reset;
  a.detach = d->detach_reset;
  a.sg = d->surrogate;
  if (d->surrogate == SNN_SG_FAST_SIGMOID) {
    a.sg_a = d->sg_param;
    a.sg_b = 0.0f;
  } else {
    a.sg_a = (float)(0.5 * (double)d->sg_param);
    a.sg_b = (float)(M_PI * 0.5 * (double)d->sg_param);
  }
  a.beta_mode = d->beta_mode;
  a.thr_mode = d->thr_mode;
  a.alpha_mode = d->alpha_mode;
  a.status = ws_view(ws, d).status;
  a.wait_ns = d->wait_limit_ns > 0 ? (uint64_t)d->wait_limit_ns : kDefaultWaitNs;
  a.debug = d->debug_flags;
  return a;
}

snn_status_t cuda_status(cudaError_t e) {
  if (e == cudaSuccess) return SNN_OK;
  if (e == cudaErrorNotSupported) return SNN_ERR_UNSUPPORTED;
  return SNN_ERR_CUDA;
}

// Neuron kinds of the shared scan paths.
enum Neuron { kLeaky = 0, kSynaptic = 1, kRecurrentLeaky = 2 };

snn_status_t scan_fwd(const snn_scan_desc* d, int neuron, const void* I, const float* alpha,
                      const float* beta, const float* thr, const float* mem0, const float* syn0,
                      void* spk, void* mem, void* synout, float* ckpt, float* mem_final,
                      float* syn_final, void* ws, size_t ws_bytes, cudaStream_t stream) {
  snn_status_t s = check_desc(d);
  if (s != SNN_OK) return s;
  const bool syn = neuron == kSynaptic, rec = neuron == kRecurrentLeaky;
  const int64_t n = d->T * d->B * d->N;
  const bool recompute = d->save == SNN_SAVE_RECOMPUTE;
  if (!beta || !thr || ((syn || rec) && !alpha)) return SNN_ERR_INVALID_ARG;
  if (rec && d->reset != SNN_RESET_SUBTRACT) return SNN_ERR_UNSUPPORTED;
  if (n > 0 && (!I || !spk)) return SNN_ERR_INVALID_ARG;
  if (n > 0 && !recompute && !mem) return SNN_ERR_INVALID_ARG;
  if (recompute && snn_scan_ckpt_elems(d, syn) > 0 && !ckpt) return SNN_ERR_INVALID_ARG;
  if ((s = check_ptrs({I, alpha, beta, thr, mem0, syn0, spk, mem, synout, ckpt, mem_final, syn_final})) != SNN_OK)
    return s;
  if ((s = check_ws(d, ws, ws_bytes)) != SNN_OK) return s;
  if (d->B * d->N == 0) return SNN_OK;
  ScanArgs a = base_args(d, ws);
  a.beta = beta;
  a.thr = thr;
  a.alpha = (syn || rec) ? alpha : nullptr;
  a.rec = rec ? 1 : 0;
  a.mem0 = mem0;
  a.syn0 = syn ? syn0 : nullptr;
  a.I = I;
  a.spk = spk;
  a.mem = mem;
  a.syn = syn ? synout : nullptr;
  a.ckpt = recompute ? ckpt : nullptr;
  const bool staged = staged_ok(d);
  if (!recompute && d->io_dtype != SNN_F32 && ckpt && staged) {
    a.bits = reinterpret_cast<unsigned char*>(ckpt);
    a.bits_row = spike_bits_row(d);
  }
  a.mem_final = mem_final;
  a.syn_final = syn ? syn_final : nullptr;
  return cuda_status(launch_scan_fwd(a, syn, d->in_dtype, d->io_dtype, staged, stream));
}

snn_status_t scan_bwd(const snn_scan_desc* d, int neuron, const void* I, const float* ckpt,
                      const void* mem, const void* spk, const void* synin, const float* alpha,
                      const float* beta, const float* thr, const float* mem0, const float* syn0,
                      const void* grad_spk, const void* grad_mem, const float* grad_mem_final,
                      const float* grad_syn_final, void* grad_I, float* grad_alpha,
                      float* grad_beta, float* grad_thr, float* grad_mem0, float* grad_syn0,
                      void* ws, size_t ws_bytes, cudaStream_t stream,
                      bool reset_control = false) {
  snn_status_t s = check_desc(d);
  if (s != SNN_OK) return s;
  const bool syn = neuron == kSynaptic, rec = neuron == kRecurrentLeaky;
  const int64_t n = d->T * d->B * d->N;
  const bool recompute = d->save == SNN_SAVE_RECOMPUTE;
  if (!beta || !thr || ((syn || rec) && !alpha)) return SNN_ERR_INVALID_ARG;
  if (rec && d->reset != SNN_RESET_SUBTRACT) return SNN_ERR_UNSUPPORTED;
  if (n > 0 && (!grad_spk || !grad_I)) return SNN_ERR_INVALID_ARG;
  if (n > 0 && recompute && !I) return SNN_ERR_INVALID_ARG;
  if (recompute && snn_scan_ckpt_elems(d, syn) > 0 && !ckpt) return SNN_ERR_INVALID_ARG;
  if (n > 0 && !recompute) {
    if (!mem) return SNN_ERR_INVALID_ARG;
    // a rounded mem cannot give back the spike: spk rows, or the bit rows
    // (which only the staged kernels read)
    if (d->io_dtype != SNN_F32 && !spk && !(ckpt && staged_ok(d))) return SNN_ERR_INVALID_ARG;
    if (syn && grad_alpha && !synin) return SNN_ERR_INVALID_ARG;
  }
  if ((s = check_ptrs({I, ckpt, mem, spk, synin, alpha, beta, thr, mem0, syn0, grad_spk, grad_mem,
                       grad_mem_final, grad_syn_final, grad_I, grad_alpha, grad_beta, grad_thr,
                       grad_mem0, grad_syn0})) != SNN_OK)
    return s;
  if ((s = check_ws(d, ws, ws_bytes)) != SNN_OK) return s;
  if (reset_control) {
    // a workspace whose previous contents are unknown (another layout, or a
    // call that gave up): zero the status word and every ticket this call's
    // reductions take, on the stream, before any kernel reads them
    const size_t tickets = kStatusBytes + 3 * lane_bytes(d) + 3 * (size_t)red_scratch(d) * sizeof(double);
    if (cudaMemsetAsync(ws, 0, kStatusBytes, stream) != cudaSuccess) return SNN_ERR_CUDA;
    if (cudaMemsetAsync(static_cast<unsigned char*>(ws) + tickets, 0, 3 * ticket_bytes(d), stream) !=
        cudaSuccess)
      return SNN_ERR_CUDA;
  }
  const int64_t L = d->B * d->N;
  float* outs[3] = {grad_beta, grad_thr, (syn || rec) ? grad_alpha : nullptr};
  const int modes[3] = {d->beta_mode, d->thr_mode, d->alpha_mode};
  if (L == 0) {
    for (int k = 0; k < 3; ++k)
      if (outs[k]) {
        cudaError_t e = cudaMemsetAsync(outs[k], 0, param_len(modes[k], d) * sizeof(float), stream);
        if (e != cudaSuccess) return SNN_ERR_CUDA;
      }
    return SNN_OK;
  }
  WsView v = ws_view(ws, d);
  ScanArgs a = base_args(d, ws);
  a.beta = beta;
  a.thr = thr;
  a.alpha = (syn || rec) ? alpha : nullptr;
  a.rec = rec ? 1 : 0;
  a.mem0 = mem0;
  a.syn0 = syn ? syn0 : nullptr;
  a.I = recompute ? I : nullptr;
  a.ckpt = recompute ? const_cast<float*>(ckpt) : nullptr;
  a.mem_in = recompute ? nullptr : mem;
  a.spk_in = (!recompute && d->io_dtype != SNN_F32) ? spk : nullptr;
  if (!recompute && d->io_dtype != SNN_F32 && ckpt && staged_ok(d)) {
    a.bits = reinterpret_cast<unsigned char*>(const_cast<float*>(ckpt));
    a.bits_row = spike_bits_row(d);
  }
  a.syn_in = (syn && !recompute && grad_alpha) ? synin : nullptr;
  a.gs = grad_spk;
  a.gm = grad_mem;
  a.gmf = grad_mem_final;
  a.gsf = syn ? grad_syn_final : nullptr;
  a.gI = grad_I;
  a.part_beta = grad_beta ? v.part[0] : nullptr;
  a.part_thr = grad_thr ? v.part[1] : nullptr;
  a.part_alpha = ((syn || rec) && grad_alpha) ? v.part[2] : nullptr;
  a.gmem0 = grad_mem0;
  a.gsyn0 = syn ? grad_syn0 : nullptr;
  const bool staged = staged_ok(d);
  cudaError_t e = syn ? launch_scan_bwd_synaptic(a, recompute, d->in_dtype, d->io_dtype, staged, stream)
                      : launch_scan_bwd_leaky(a, recompute, d->in_dtype, d->io_dtype, staged, stream);
  if (e != cudaSuccess) return cuda_status(e);
  // one launch per parameter layout in use
  float* parts[3] = {a.part_beta, a.part_thr, a.part_alpha};
  for (int mode = SNN_P_SCALAR; mode <= SNN_P_PER_CHANNEL; ++mode) {
    ParamReduce jobs[3];
    int n = 0;
    for (int k = 0; k < 3; ++k)
      if (outs[k] && modes[k] == mode) jobs[n++] = ParamReduce{parts[k], outs[k], v.scratch[k], v.tickets[k]};
    if (n == 0) continue;
    e = launch_param_reduce(jobs, n, d->B, d->N, d->C, d->HW, mode, red_scratch(d), stream);
    if (e != cudaSuccess) return SNN_ERR_CUDA;
  }
  return SNN_OK;
}

}  // namespace

std::atomic<unsigned long long> g_kernel_launches{0};

// snn_leaky_bwd on a workspace whose contents are left over from earlier
// calls of any layout: after the argument checks, the status word and the
// reductions' tickets are zeroed on the stream (snn_noalloc.cu).
snn_status_t leaky_bwd_reset_workspace(const snn_scan_desc* d, const void* I, const float* ckpt,
                                       const void* mem, const void* spk, const float* beta,
                                       const float* thr, const float* mem0, const void* grad_spk,
                                       const void* grad_mem, const float* grad_mem_final,
                                       void* grad_I, float* grad_beta, float* grad_thr,
                                       float* grad_mem0, void* ws, size_t ws_bytes,
                                       cudaStream_t stream) {
  return scan_bwd(d, kLeaky, I, ckpt, mem, spk, nullptr, nullptr, beta, thr, mem0, nullptr,
                  grad_spk, grad_mem, grad_mem_final, nullptr, grad_I, nullptr, grad_beta,
                  grad_thr, grad_mem0, nullptr, ws, ws_bytes, stream, true);
}

}  // namespace snn

using namespace snn;

extern "C" {

uint64_t snn_kernel_launches(void) { return g_kernel_launches.load(std::memory_order_relaxed); }

const char* snn_status_string(snn_status_t status) {
  switch (status) {
    case SNN_OK: return "SNN_OK";
    case SNN_ERR_INVALID_ARG: return "SNN_ERR_INVALID_ARG: invalid or inconsistent argument";
    case SNN_ERR_ALIGNMENT: return "SNN_ERR_ALIGNMENT: a device pointer is not 16-byte aligned";
    case SNN_ERR_UNSUPPORTED: return "SNN_ERR_UNSUPPORTED: combination not implemented";
    case SNN_ERR_WORKSPACE: return "SNN_ERR_WORKSPACE: workspace missing or too small";
    case SNN_ERR_CUDA: return "SNN_ERR_CUDA: CUDA runtime error";
    case SNN_ERR_TIMEOUT: return "SNN_ERR_TIMEOUT: an in-kernel wait gave up";
  }
  return "SNN_ERR_UNKNOWN: unknown status code";
}

int snn_version(void) { return 100; }

size_t snn_scan_desc_size(void) { return sizeof(snn_scan_desc); }

size_t snn_scan_workspace_bytes(const snn_scan_desc* desc) {
  if (check_desc(desc) != SNN_OK) return 0;
  return workspace_bytes(desc);
}

int64_t snn_scan_ckpt_elems(const snn_scan_desc* desc, int synaptic) {
  if (check_desc(desc) != SNN_OK) return 0;
  if (desc->save != SNN_SAVE_RECOMPUTE) {
    if (desc->io_dtype == SNN_F32) return 0;
    return desc->T * spike_bits_row(desc) / 4;  // spike bits, in fp32 units
  }
  const int64_t nseg = ceil_div(desc->T, desc->ckpt_every);
  const int64_t n = nseg > 1 ? (nseg - 1) * desc->B * desc->N : 0;
  return synaptic ? 2 * n : n;
}

snn_status_t snn_workspace_init(void* ws, size_t ws_bytes, snn_stream_t stream) {
  if (!ws || ws_bytes < kStatusBytes) return SNN_ERR_WORKSPACE;
  if (!aligned16(ws)) return SNN_ERR_ALIGNMENT;
  return cudaMemsetAsync(ws, 0, ws_bytes, (cudaStream_t)stream) == cudaSuccess ? SNN_OK : SNN_ERR_CUDA;
}

snn_status_t snn_workspace_status(void* ws, snn_stream_t stream) {
  if (!ws) return SNN_ERR_WORKSPACE;
  if (!aligned16(ws)) return SNN_ERR_ALIGNMENT;
  int host = 0;
  cudaStream_t st = (cudaStream_t)stream;
  if (cudaMemcpyAsync(&host, ws, sizeof(int), cudaMemcpyDeviceToHost, st) != cudaSuccess) return SNN_ERR_CUDA;
  if (cudaMemsetAsync(ws, 0, sizeof(int), st) != cudaSuccess) return SNN_ERR_CUDA;
  if (cudaStreamSynchronize(st) != cudaSuccess) return SNN_ERR_CUDA;
  return (snn_status_t)host;
}

snn_status_t snn_leaky_fwd(const snn_scan_desc* desc, const void* I, const float* beta,
                           const float* thr, const float* mem0, void* spk, void* mem,
                           float* ckpt, float* mem_final, void* ws, size_t ws_bytes,
                           snn_stream_t stream) {
  return scan_fwd(desc, kLeaky, I, nullptr, beta, thr, mem0, nullptr, spk, mem, nullptr, ckpt,
                  mem_final, nullptr, ws, ws_bytes, (cudaStream_t)stream);
}

snn_status_t snn_leaky_bwd(const snn_scan_desc* desc, const void* I, const float* ckpt,
                           const void* mem, const void* spk, const float* beta,
                           const float* thr, const float* mem0, const void* grad_spk,
                           const void* grad_mem, const float* grad_mem_final, void* grad_I,
                           float* grad_beta, float* grad_thr, float* grad_mem0, void* ws,
                           size_t ws_bytes, snn_stream_t stream) {
  return scan_bwd(desc, kLeaky, I, ckpt, mem, spk, nullptr, nullptr, beta, thr, mem0, nullptr,
                  grad_spk, grad_mem, grad_mem_final, nullptr, grad_I, nullptr, grad_beta,
                  grad_thr, grad_mem0, nullptr, ws, ws_bytes, (cudaStream_t)stream);
}

snn_status_t snn_synaptic_fwd(const snn_scan_desc* desc, const void* I, const float* alpha,
                              const float* beta, const float* thr, const float* mem0,
                              const float* syn0, void* spk, void* mem, void* syn,
                              float* ckpt, float* mem_final, float* syn_final, void* ws,
                              size_t ws_bytes, snn_stream_t stream) {
  return scan_fwd(desc, kSynaptic, I, alpha, beta, thr, mem0, syn0, spk, mem, syn, ckpt, mem_final,
                  syn_final, ws, ws_bytes, (cudaStream_t)stream);
}

snn_status_t snn_synaptic_bwd(const snn_scan_desc* desc, const void* I, const float* ckpt,
                              const void* mem, const void* spk, const void* syn,
                              const float* alpha, const float* beta, const float* thr,
                              const float* mem0, const float* syn0, const void* grad_spk,
                              const void* grad_mem, const float* grad_mem_final,
                              const float* grad_syn_final, void* grad_I, float* grad_alpha,
                              float* grad_beta, float* grad_thr, float* grad_mem0,
                              float* grad_syn0, void* ws, size_t ws_bytes,
                              snn_stream_t stream) {
  return scan_bwd(desc, kSynaptic, I, ckpt, mem, spk, syn, alpha, beta, thr, mem0, syn0, grad_spk,
                  grad_mem, grad_mem_final, grad_syn_final, grad_I, grad_alpha, grad_beta,
                  grad_thr, grad_mem0, grad_syn0, ws, ws_bytes, (cudaStream_t)stream);
}

snn_status_t snn_rleaky_fwd(const snn_scan_desc* desc, const void* I, const float* v,
                            const float* beta, const float* thr, const float* mem0, void* spk,
                            void* mem, float* ckpt, float* mem_final, void* ws, size_t ws_bytes,
                            snn_stream_t stream) {
  return scan_fwd(desc, kRecurrentLeaky, I, v, beta, thr, mem0, nullptr, spk, mem, nullptr, ckpt,
                  mem_final, nullptr, ws, ws_bytes, (cudaStream_t)stream);
}

snn_status_t snn_rleaky_bwd(const snn_scan_desc* desc, const void* I, const float* ckpt,
                            const void* mem, const void* spk, const float* v, const float* beta,
                            const float* thr, const float* mem0, const void* grad_spk,
                            const void* grad_mem, const float* grad_mem_final, void* grad_I,
                            float* grad_v, float* grad_beta, float* grad_thr, float* grad_mem0,
                            void* ws, size_t ws_bytes, snn_stream_t stream) {
  return scan_bwd(desc, kRecurrentLeaky, I, ckpt, mem, spk, nullptr, v, beta, thr, mem0, nullptr,
                  grad_spk, grad_mem, grad_mem_final, nullptr, grad_I, grad_v, grad_beta,
                  grad_thr, grad_mem0, nullptr, ws, ws_bytes, (cudaStream_t)stream);
}

}  // extern "C"
