// Programmatic dependent launch for the library's kernel pipelines (internal).
//
// The simulators issue a dozen or more short kernels per segment, each depending on the one
// before.  Launched as programmatic dependents, a kernel's launch and block setup overlap
// the end of its predecessor instead of following it:
//   - every kernel launched with launch_pdl() calls pdl_entry() before it touches global
//     memory: griddepcontrol.wait returns once the previous grid in the stream has completed
//     and its writes are visible;
//   - no kernel triggers its dependents early, so the next launch is scheduled when this
//     grid's blocks have exited: an earlier trigger let the dependents' blocks crowd onto
//     the SMs that freed first and made the per-sample kernels slower;
//   - dependencies that are not on a kernel of the same stream (event waits, copies) stay
//     full dependencies.
// In a kernel launched without the attribute, the wait returns at once.
#pragma once

#include <cuda_runtime.h>

#include <utility>

namespace gem {

__device__ __forceinline__ void pdl_entry() {
  asm volatile("griddepcontrol.wait;" ::: "memory");
}

template <typename... KArgs, typename... Args>
cudaError_t launch_pdl(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem,
                       cudaStream_t stream, Args&&... args) {
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
  return cudaLaunchKernelEx(&cfg, kernel, std::forward<Args>(args)...);
}

}  // namespace gem
