// Host-side launch planning shared by the scan translation units.
#pragma once

#include <cuda_runtime.h>

#include <map>
#include <mutex>
#include <tuple>

#include "scan_kernels.cuh"

namespace snn {

inline int64_t ceil_div(int64_t a, int64_t b) { return (a + b - 1) / b; }
inline int64_t round_up(int64_t a, int64_t b) { return ceil_div(a, b) * b; }

struct DeviceInfo {
  int sms = 0;
  int smem_per_sm = 0;
  int smem_optin = 0;
};

inline cudaError_t device_info(DeviceInfo* out) {
  static std::mutex mu;
  static std::map<int, DeviceInfo> cache;
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  std::lock_guard<std::mutex> g(mu);
  auto it = cache.find(dev);
  if (it != cache.end()) {
    *out = it->second;
    return cudaSuccess;
  }
  DeviceInfo d;
  if ((e = cudaDeviceGetAttribute(&d.sms, cudaDevAttrMultiProcessorCount, dev)) != cudaSuccess) return e;
  if ((e = cudaDeviceGetAttribute(&d.smem_per_sm, cudaDevAttrMaxSharedMemoryPerMultiprocessor, dev)) != cudaSuccess)
    return e;
  if ((e = cudaDeviceGetAttribute(&d.smem_optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev)) != cudaSuccess)
    return e;
  cache[dev] = d;
  *out = d;
  return cudaSuccess;
}

// Raise a kernel's dynamic shared-memory limit once per (device, kernel).
inline cudaError_t ensure_smem(const void* kernel, size_t bytes) {
  static std::mutex mu;
  static std::map<std::pair<int, const void*>, size_t> done;
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  std::lock_guard<std::mutex> g(mu);
  size_t& cur = done[{dev, kernel}];
  if (bytes <= cur || bytes <= 48 * 1024) return cudaSuccess;
  e = cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)bytes);
  if (e == cudaSuccess) cur = bytes;
  return e;
}

struct StagedPlan {
  int lanes_per_cta = 0;
  int threads = 0;  // consumer warps * 32 + one producer warp
  int stages = 0;
  int stage_bytes = 0;
  size_t smem = 0;
  int64_t grid = 0;
};

// Choose a staged launch for L lanes: all CTAs of a wave resident at once
// (grid = SMs x CTAs-per-SM x waves, lanes split evenly, strip a multiple of
// 8 lanes so every row copy starts 16-byte aligned), the deepest ring that
// fits next to the per-thread replay buffer.  Returns false if nothing fits.
//   stage_bytes_per_lane: bytes one lane contributes to the largest item
//   seg_bytes_per_thread: replay buffer bytes per consumer thread
//   lanes_per_thread: lanes each consumer thread owns
//   fixed_bytes_per_lane: other shared memory per lane of the strip
//   force_stages: exact ring depth the kernel was compiled for (0 = any)
//   max_cps: most CTAs per SM to try (larger strips first when 1)
inline bool plan_staged(const void* kernel, int64_t L, int64_t items, int stage_bytes_per_lane,
                        int seg_bytes_per_thread, int lanes_per_thread, StagedPlan* plan,
                        int fixed_bytes_per_lane = 0, int force_stages = 0, int max_cps = 2) {
  static std::mutex mu;
  static std::map<std::tuple<int, const void*, int64_t, int64_t, int, int>, StagedPlan> cache;
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return false;
  const auto key = std::make_tuple(dev, kernel, L, items, stage_bytes_per_lane,
                                   ((seg_bytes_per_thread * 64 + fixed_bytes_per_lane) * 64 +
                                    force_stages) * 4 + max_cps);
  {
    std::lock_guard<std::mutex> g(mu);
    auto it = cache.find(key);
    if (it != cache.end()) {
      *plan = it->second;
      return true;
    }
  }
  DeviceInfo d;
  if (device_info(&d) != cudaSuccess) return false;
  cudaFuncAttributes fa;
  if (cudaFuncGetAttributes(&fa, kernel) != cudaSuccess) return false;
  const int min_stages = (int)(items < 3 ? (items < 1 ? 1 : items) : 3);
  for (int waves = 1; waves <= 64; ++waves) {
    for (int cps = max_cps; cps >= 1; --cps) {
      const int64_t ctas = (int64_t)d.sms * cps * waves;
      const int64_t lpc = round_up(ceil_div(L, ctas), 8);
      const int64_t cthreads = round_up(ceil_div(lpc, lanes_per_thread), 32);
      const int threads = (int)cthreads + 32;
      if (threads > kMaxStagedThreads) continue;
      if ((int64_t)threads * fa.numRegs * cps > 65536) continue;
      const int64_t stage_bytes = round_up(lpc * stage_bytes_per_lane, 128);
      const int64_t seg_bytes = cthreads * seg_bytes_per_thread + lpc * fixed_bytes_per_lane;
      const int64_t budget = (int64_t)d.smem_per_sm / cps - 1024 - (int64_t)fa.sharedSizeBytes;
      const int64_t avail = (budget < d.smem_optin ? budget : d.smem_optin) - kBarrierBytes - seg_bytes;
      if (avail < stage_bytes * (force_stages > 0 ? force_stages : min_stages)) continue;
      int64_t stages = avail / stage_bytes;
      if (stages > kMaxStages) stages = kMaxStages;
      if (stages > items && items > 0) stages = items;
      if (stages < 1) stages = 1;
      if (force_stages > 0) stages = force_stages;
      StagedPlan p;
      p.lanes_per_cta = (int)lpc;
      p.threads = threads;
      p.stages = (int)stages;
      p.stage_bytes = (int)stage_bytes;
      p.smem = (size_t)(kBarrierBytes + stages * stage_bytes + seg_bytes);
      p.grid = ceil_div(L, lpc);
      if (ensure_smem(kernel, p.smem) != cudaSuccess) continue;
      int nb = 0;
      if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&nb, kernel, threads, p.smem) != cudaSuccess)
        continue;
      if (nb < cps) continue;
      std::lock_guard<std::mutex> g(mu);
      cache[key] = p;
      *plan = p;
      return true;
    }
  }
  return false;
}

// Entry points of the per-translation-unit dispatchers.  dtype codes follow
// snn_dtype_t; `staged` selects the TMA-staged kernels (the caller checked
// row alignment).  Return cudaErrorNotSupported for a combination that is
// not instantiated.
cudaError_t launch_scan_fwd(ScanArgs a, bool synaptic, int in_dt, int io_dt, bool staged,
                            cudaStream_t stream);
cudaError_t launch_scan_bwd_leaky(ScanArgs a, bool recompute, int in_dt, int io_dt, bool staged,
                                  cudaStream_t stream);
cudaError_t launch_scan_bwd_synaptic(ScanArgs a, bool recompute, int in_dt, int io_dt,
                                     bool staged, cudaStream_t stream);
// the recompute variants, compiled in translation units of their own
cudaError_t launch_scan_bwd_leaky_recompute(ScanArgs a, int in_dt, int io_dt, bool staged,
                                            cudaStream_t stream);
cudaError_t launch_scan_bwd_synaptic_recompute(ScanArgs a, int in_dt, int io_dt, bool staged,
                                               cudaStream_t stream);
// the recompute BPTT of the Leaky neuron with the replayed segment in
// registers (scan_bwd_seg), for checkpoint intervals 8, 12 and 16; sets
// *launched, and launches nothing where it does not apply
cudaError_t launch_scan_bwd_leaky_seg(ScanArgs a, int in_dt, int io_dt, bool staged,
                                      cudaStream_t stream, bool* launched);
// fp64 scratch the reduction of one parameter needs (elements)
inline int64_t param_reduce_scratch(int64_t N, int64_t C) {
  const int64_t a = 1024, b = 8 * N, c = 64 * C;
  return a > b ? (a > c ? a : c) : (b > c ? b : c);
}
// One parameter's reduction: per-lane partials in, gradient out, fp64
// scratch and zero-initialised tickets (one per output group: 1 for a
// scalar, C per channel; the per-neuron reduction needs neither, the
// workspace keeps ceil(N/256) slots for it) from the workspace.
struct ParamReduce {
  const float* part;
  float* out;
  double* scratch;
  int* tickets;
};
inline int64_t param_reduce_groups(int64_t N, int64_t C) {
  const int64_t a = (N + 255) / 256;
  return a > C ? (a > 1 ? a : 1) : (C > 1 ? C : 1);
}
// Reduce n (<= 3) parameters that share `mode` in one launch.
cudaError_t launch_param_reduce(const ParamReduce* p, int n, int64_t B, int64_t N, int64_t C,
                                int64_t HW, int mode, int64_t scratch_len, cudaStream_t stream);

}  // namespace snn
