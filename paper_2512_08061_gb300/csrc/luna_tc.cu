// Tensor-core (tcgen05 / TMEM / TMA) path for bf16 I/O on sm_103a.
#include "luna_tc.cuh"

namespace luna {

TcPlan tc_plan(const luna_attn_desc &, const TableLayout &) { return TcPlan{}; }

bool tc_inputs_ok(const TcPlan &, const void *, const void *, const void *, const void *) { return false; }

cudaError_t launch_tc_fwd(const TcPlan &, const AttnArgs &, char *, cudaStream_t) { return cudaErrorNotSupported; }

cudaError_t launch_tc_bwd(const TcPlan &, const AttnArgs &, char *, bool, cudaStream_t) {
    return cudaErrorNotSupported;
}

}  // namespace luna
