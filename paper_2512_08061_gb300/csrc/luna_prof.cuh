// Kernel timing hook (see luna_profile_start in luna.h) and the launch macros.
#pragma once

#include <utility>

#include "luna_common.cuh"

namespace luna {

void prof_before(const char *kernel, cudaStream_t s);  // also counts the launch
void prof_after(const char *kernel, cudaStream_t s);

// Launches `kernel` bracketed by the timing hook under the name `tag`.
#define LUNA_LAUNCH(tag, kernel, grid, block, smem, stream, ...)  \
    do {                                                          \
        ::luna::prof_before(tag, stream);                         \
        kernel<<<grid, block, smem, stream>>>(__VA_ARGS__);        \
        ::luna::prof_after(tag, stream);                          \
    } while (0)

// Programmatic dependent launch.  With `dep` set, the kernel may be scheduled
// before the previous kernel of the stream has finished: its blocks start as
// that kernel's blocks leave the SMs, run their prologue, and reach the
// previous kernel's results only through grid_dependency_sync().  Every kernel
// launched this way calls grid_dependency_sync() in every block, before it
// reads anything a kernel of the same stream may still be writing (anything
// but the parameter table, which the calls that use this launch never write
// after their first cudaMemsetAsync) and before its first global store;
// since each block waits there, the stream's order stays transitive.
template <typename... KArgs, typename... Args>
cudaError_t launch_dep(bool dep, void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t s,
                       Args &&...args) {
    cudaLaunchAttribute at[1];
    at[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    at[0].val.programmaticStreamSerializationAllowed = 1;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = grid;
    cfg.blockDim = block;
    cfg.dynamicSmemBytes = smem;
    cfg.stream = s;
    cfg.attrs = at;
    cfg.numAttrs = dep ? 1 : 0;
    return cudaLaunchKernelEx(&cfg, kernel, std::forward<Args>(args)...);
}

#define LUNA_LAUNCH_DEP(tag, dep, kernel, grid, block, smem, stream, ...)           \
    do {                                                                           \
        ::luna::prof_before(tag, stream);                                          \
        (void)::luna::launch_dep(dep, kernel, grid, block, smem, stream, __VA_ARGS__); \
        ::luna::prof_after(tag, stream);                                           \
    } while (0)

#ifdef __CUDACC__
// Waits until the grids this one depends on have completed and their memory
// is visible (at once when the launch had no programmatic dependency), then
// lets the next kernel of the stream be scheduled.  Every thread of the block
// calls it.
__device__ __forceinline__ void grid_dependency_sync() {
    asm volatile("griddepcontrol.wait;" ::: "memory");
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}
#endif

}  // namespace luna
