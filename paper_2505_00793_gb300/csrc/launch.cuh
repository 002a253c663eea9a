// Kernel launches with programmatic dependent launch (PDL).
//
// Every kernel of the library starts with pdl_entry(): it waits until the previous kernel on
// the stream has completed and its writes are visible (griddepcontrol.wait), then lets the
// next kernel on the stream begin launching (griddepcontrol.launch_dependents).  Launched
// with the programmatic-serialization attribute, a kernel's launch, CTA rasterisation and
// prologue (barrier init, TMEM allocation, tensor-map prefetch) overlap the tail of its
// predecessor; nothing it reads or writes in global memory is touched before the wait, so
// the stream order of memory effects is unchanged.  The wait is a no-op for a kernel
// launched without the attribute, so both launch forms are correct.
#pragma once

#include <cuda_runtime.h>

#include <utility>

namespace mf {

// Process-wide switch (mf_set_option MF_OPT_PDL); 1 = launch with the attribute.
extern int g_pdl;

__device__ __forceinline__ void pdl_wait() {
  asm volatile("griddepcontrol.wait;" ::: "memory");
}
__device__ __forceinline__ void pdl_trigger() {
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}
__device__ __forceinline__ void pdl_entry() {
  pdl_wait();
  pdl_trigger();
}

template <typename... KArgs, typename... Args>
cudaError_t launch_k(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem,
                     cudaStream_t s, Args&&... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = g_pdl ? 1 : 0;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kernel, std::forward<Args>(args)...);
}

}  // namespace mf
