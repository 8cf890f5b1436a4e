// Programmatic dependent launch.  A kernel launched with launch_pdl may be
// scheduled while the kernel before it on the stream is still running, so
// its launch latency overlaps that kernel's tail.  Such a kernel calls
// pdl_wait() before it touches memory the earlier kernels write or read
// (griddepcontrol.wait returns once they have completed and their writes are
// visible), and pdl_trigger() to let the next kernel be scheduled early.
// Both are no-ops for kernels launched the ordinary way.
#pragma once
#include <cuda_runtime.h>

#include <utility>

namespace fasgd {

__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void pdl_trigger() { asm volatile("griddepcontrol.launch_dependents;" ::: "memory"); }

template <typename... Exp, typename... Act>
cudaError_t launch_pdl(void (*kernel)(Exp...), dim3 grid, dim3 block, size_t smem,
                       cudaStream_t stream, Act&&... args) {
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
    return cudaLaunchKernelEx(&cfg, kernel, std::forward<Act>(args)...);
}

}  // namespace fasgd
