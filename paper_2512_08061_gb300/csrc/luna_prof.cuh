// Kernel timing hook (see luna_profile_start in luna.h).
#pragma once

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

}  // namespace luna
