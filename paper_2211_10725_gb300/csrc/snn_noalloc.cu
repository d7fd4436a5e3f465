// Leaky BPTT for callers that cannot allocate device memory.
//
// snn_leaky_bwd needs a caller-provided workspace (a status word, per-lane
// parameter-gradient partials and reduction scratch).  Some callers cannot
// allocate one: hosts that do not own the device allocator (memory is
// budgeted up front by another runtime), real-time loops that must not call
// cudaMalloc because it can synchronise the device, or plain C hosts with no
// allocator at all.  snn_leaky_bwd_noalloc runs the same computation with its
// scratch in a fixed array in the library's own device memory instead.
//
// The array is a file-scope __device__ variable: every GPU that loads the
// library holds kNoAllocScratchBytes of it until the process exits.  Host
// code must not use its name as an address (that is a host-side stand-in);
// the device address is looked up once per device with
// cudaGetSymbolAddress, while that device is current.
#include <cstdint>
#include <map>
#include <mutex>

#include <cuda_runtime.h>

#include "snn.h"

namespace {

// Largest workspace (snn_scan_workspace_bytes) the entry point serves.
constexpr size_t kNoAllocScratchBytes = size_t(16) << 20;

static __device__ __align__(256) unsigned char g_noalloc_scratch[kNoAllocScratchBytes];

// Device address of g_noalloc_scratch on the current device; the first call
// on a device looks it up (not a stream operation) and caches it.
cudaError_t scratch_address(void** out) {
  static std::mutex mu;
  static std::map<int, void*> cache;
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  std::lock_guard<std::mutex> g(mu);
  auto it = cache.find(dev);
  if (it != cache.end()) {
    *out = it->second;
    return cudaSuccess;
  }
  void* p = nullptr;
  e = cudaGetSymbolAddress(&p, g_noalloc_scratch);
  if (e != cudaSuccess) return e;
  cache[dev] = p;
  *out = p;
  return cudaSuccess;
}

}  // namespace

namespace snn {
// snn_leaky_bwd that first zeroes the workspace's status word and the
// tickets of this call's reductions (snn_api.cu).
snn_status_t leaky_bwd_reset_workspace(const snn_scan_desc* d, const void* I, const float* ckpt,
                                       const void* mem, const void* spk, const float* beta,
                                       const float* thr, const float* mem0, const void* grad_spk,
                                       const void* grad_mem, const float* grad_mem_final,
                                       void* grad_I, float* grad_beta, float* grad_thr,
                                       float* grad_mem0, void* ws, size_t ws_bytes,
                                       cudaStream_t stream);
}  // namespace snn

extern "C" snn_status_t snn_leaky_bwd_noalloc(
    const snn_scan_desc* desc, const void* I, const float* ckpt, const void* mem,
    const void* spk, const float* beta, const float* thr, const float* mem0,
    const void* grad_spk, const void* grad_mem, const float* grad_mem_final, void* grad_I,
    float* grad_beta, float* grad_thr, float* grad_mem0, int* status, snn_stream_t stream) {
  if (status && (reinterpret_cast<uintptr_t>(status) & 3u) != 0) return SNN_ERR_ALIGNMENT;
  void* ws = nullptr;
  if (scratch_address(&ws) != cudaSuccess) return SNN_ERR_CUDA;
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  // The scratch keeps whatever the previous call left: another layout (its
  // tickets sit at offsets that depend on B, N and C), or the leftovers of a
  // call that timed out.  After the same argument checks as snn_leaky_bwd
  // (a workspace beyond kNoAllocScratchBytes fails them with
  // SNN_ERR_WORKSPACE), the status word and every reduction ticket this call
  // takes are zeroed on the stream; the partials and the fp64 scratch are
  // written by this call before they are read.
  const snn_status_t s = snn::leaky_bwd_reset_workspace(
      desc, I, ckpt, mem, spk, beta, thr, mem0, grad_spk, grad_mem, grad_mem_final, grad_I,
      grad_beta, grad_thr, grad_mem0, ws, kNoAllocScratchBytes, st);
  if (s != SNN_OK) return s;
  if (status &&
      cudaMemcpyAsync(status, ws, sizeof(int), cudaMemcpyDeviceToDevice, st) != cudaSuccess)
    return SNN_ERR_CUDA;
  return SNN_OK;
}
