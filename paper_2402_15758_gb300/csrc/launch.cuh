// Kernel launches with programmatic stream serialization: a kernel may begin launching
// while its predecessor in the stream drains; every kernel of the library calls
// pdl_wait() before it touches memory written by earlier kernels.  No kernel parameter
// is `const T* __restrict__`: the compiler may treat loads through such a pointer as
// invariant for the whole kernel and schedule them ahead of the wait.
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
