// Kernel launches with programmatic dependent launch: a kernel may be
// scheduled while the kernel before it on the stream is still retiring, and
// runs its set-up (barrier initialisation, tensor-memory allocation) in that
// time.  Every kernel calls grid_dep_wait() before its first global-memory
// access, which returns once the preceding grid has completed and its
// writes are visible, so stream order is kept for all data.
#pragma once

#include <cuda_runtime.h>

#include <atomic>

namespace snn {

// Kernels launched (or captured into a graph) through launch_pdl in this
// process; read through snn_kernel_launches().
extern std::atomic<unsigned long long> g_kernel_launches;

__device__ __forceinline__ void grid_dep_wait() {
  asm volatile("griddepcontrol.wait;" ::: "memory");
}

template <typename... Params, typename... Args>
cudaError_t launch_pdl(void (*kernel)(Params...), dim3 grid, dim3 block, size_t smem,
                       cudaStream_t stream, Args... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  const cudaError_t e = cudaLaunchKernelEx(&cfg, kernel, static_cast<Params>(args)...);
  if (e == cudaSuccess) g_kernel_launches.fetch_add(1, std::memory_order_relaxed);
  return e;
}

}  // namespace snn
