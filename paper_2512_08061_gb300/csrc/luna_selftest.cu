// Exercise of the failure path of the bounded device waits: one block waits on
// an mbarrier phase that nothing completes, gives up after `limit_ns` of wall
// time (%globaltimer), and reports through the status word of the workspace
// exactly as a kernel whose wait ran out does.  The kernel always ends.
#include "luna_prof.cuh"
#include "luna_sm100.cuh"
#include "luna_simt.cuh"

namespace luna {
namespace {

__global__ void __launch_bounds__(32) k_selftest_wait(int *status, unsigned long long limit_ns) {
    __shared__ uint64_t bar;
    if (threadIdx.x == 0) {
        sm100::mbar_init(&bar, 1);  // expects one arrival that never comes
        sm100::fence_mbar_init();
    }
    __syncwarp();
    if (threadIdx.x == 0 && !sm100::mbar_wait(&bar, 0, limit_ns)) atomicOr(status, 1);
}

}  // namespace

cudaError_t launch_selftest_wait(int *status, long long limit_ns, cudaStream_t s) {
    LUNA_LAUNCH("selftest_wait", k_selftest_wait, 1, 32, 0, s, status, (unsigned long long)limit_ns);
    return cudaGetLastError();
}

}  // namespace luna
