// Programmatic dependent launch between the library's kernels.
//
// Every kernel of the revisit path is launched with programmatic stream
// serialization. It allows its dependents at entry, so the next kernel's CTAs
// may be launched as soon as every CTA of this grid is resident. Before its
// first global load or store it waits for the grid it depends on to complete
// and its writes to be visible. Only L2 prefetches, which return nothing to
// the thread, go before that wait. A kernel whose predecessor is not one of
// these (it never allows dependents) is launched when the predecessor
// completes, as with a plain launch, and its wait returns at once.
#pragma once

#include <utility>

#include <cuda_runtime.h>

namespace prcr {

__device__ __forceinline__ void pdl_allow() {
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}

__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }

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

}  // namespace prcr
