// Tensor-core (tcgen05 / TMEM / TMA) path for bf16 I/O on sm_103a.
#pragma once

#include "luna_simt.cuh"

namespace luna {

struct TcPlan {
    bool eligible = false;   // shape and dtype handled by the tensor-core kernels
    int variant = -1;        // kernel instantiation (value width / projections)
    bool bwd = false;        // backward also on tensor cores
    bool causal_fwd = false; // streaming-form forward on tensor cores
    bool causal_bwd = false; // streaming-form backward on tensor cores
    size_t ws_fwd = 0, ws_bwd = 0;
};

TcPlan tc_plan(const luna_attn_desc &ad, const TableLayout &lay);
bool tc_inputs_ok(const TcPlan &p, const void *a, const void *b, const void *c, const void *d);
cudaError_t launch_tc_fwd(const TcPlan &p, const AttnArgs &a, char *ws, cudaStream_t s);
cudaError_t launch_tc_bwd(const TcPlan &p, const AttnArgs &a, char *ws, bool have_stats, cudaStream_t s);
cudaError_t launch_tc_stats(const AttnArgs &a, cudaStream_t s);
// Work items of the persistent non-causal kernels (chunks of whole 128-row tiles of one head) and, for
// padded sequences, their split over the grid balanced by valid tiles (a small split kernel on s).
// zmask: outputs whose padded rows the split launch zeroes (1: O, 2: dQ, 4: dK, 8: dV).
AttnArgs tc_balanced_items(const AttnArgs &a, cudaStream_t s, cudaError_t *err, int zmask);
int tc_grid(const AttnArgs &items);  // persistent grid of the non-causal kernels
constexpr int kMaxGrid = 1024;       // split entries the workspace holds
bool tc_bwd_supported(const luna_attn_desc &ad, const TableLayout &lay);
bool tc_bwd_fits(const AttnArgs &a);
cudaError_t launch_tc_bwd_kernels(const AttnArgs &a, bool have_stats, cudaStream_t s);
cudaError_t launch_tc_bwd_wide(const AttnArgs &a, bool have_stats, cudaStream_t s);  // d = dv = 64
// key statistics of every work item (a.rows_per_split rows, a.nsplit per head) into S_part, z_part
cudaError_t launch_tc_keys_items(const AttnArgs &a, cudaStream_t s);
bool tc_causal_supported(const luna_attn_desc &ad, const TableLayout &lay);
cudaError_t launch_tc_causal_fwd(const AttnArgs &a, cudaStream_t s);
// segment prefixes of S, z (work items = state segments)
cudaError_t launch_tc_causal_stats(const AttnArgs &a, cudaStream_t s);
cudaError_t launch_tc_causal_bwd(const AttnArgs &a, bool have_state, cudaStream_t s);

}  // namespace luna
