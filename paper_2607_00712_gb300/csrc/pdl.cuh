// Programmatic dependent launch between kernels that follow each other on one stream: a
// kernel launched with launch_pdl may start (and run its prologue: barrier set-up, TMEM
// allocation) while the kernel before it finishes; it calls pdl_wait() before its first
// access to global memory that the earlier kernel may write (or, for a write of its own, may
// still read), which returns once that kernel has completed and its writes are visible.  pdl_trigger() in the earlier kernel lets the
// dependent start before all of its blocks have exited.
#pragma once

#include <cuda_runtime.h>

#include <utility>

namespace ispa {

__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void pdl_trigger() { asm volatile("griddepcontrol.launch_dependents;" ::: "memory"); }

template <typename... KArgs, typename... Args>
cudaError_t launch_pdl(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t s,
                       Args&&... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kernel, std::forward<Args>(args)...);
}

}  // namespace ispa
