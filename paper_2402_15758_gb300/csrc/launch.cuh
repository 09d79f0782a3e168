// Kernel launches with programmatic stream serialization: a kernel may begin launching
// while its predecessor in the stream drains.  Every kernel calls pdl_wait() before it
// touches memory written by earlier kernels, with one exception: the tensor-core tree
// attention with prewait_kv set reads n_ctx, the page table and committed KV rows
// before its wait.  That is correct only because the launch directly before it is a
// tensor-core linear, which lets dependents launch only after its own pdl_wait (so
// every earlier kernel is complete); the row kernels trigger before they wait, and the
// runtime refuses to enqueue such an attention after anything but a tensor-core
// linear.  No kernel parameter is `const T* __restrict__`: the compiler may treat loads
// through such a pointer as invariant for the whole kernel and schedule them ahead of
// the wait.
#pragma once

#include <cuda_runtime.h>

namespace chimera {

template <typename... KArgs, typename... Args>
inline cudaError_t launch_pdl(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t s,
                              Args&&... args) {
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kernel, std::forward<Args>(args)...);
}

}  // namespace chimera
