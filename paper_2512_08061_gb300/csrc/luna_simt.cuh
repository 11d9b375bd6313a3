// Launch arguments and entry points of the generic (CUDA-core, fp32) kernels.
#pragma once

#include "luna_common.cuh"

namespace luna {

struct AttnArgs {
    int B, H, n, d, dv, M, L, D;
    float eps;
    TableLayout lay;
    const char *table;
    const void *Q, *K, *V, *dO;
    void *O, *dQ, *dK, *dV;
    const int32_t *lengths;
    // non-causal statistics
    int nsplit, rows_per_split;        // key-statistics splits per head
    float *S_part, *z_part;            // [BH][nsplit][D][dv], [BH][nsplit][D]
    float *S_fin, *z_fin;              // [BH][D][dv], [BH][D]
    int *counters;                     // [2*BH], zero on entry
    // backward
    int nsplit_b, rows_per_split_b;
    float *dS_part, *dz_part, *dS_fin, *dz_fin;
    float *gpart;                      // [2 * BH * nsplit_b][gsize] parameter-gradient partials (fp32, or
                                       // fp64 when gpart64: the generic kernels)
    int gpart64;                       // 1: the partials are doubles
    int gsize;                         // M*d + M + nint*L*2
    double *hist;                      // [gsize] the partials' sum: dW, db, then the histogram [nint][L][2]
    luna_phi_grads grads;
    // causal
    int chunk, seg_len, nseg;          // state segments of seg_len rows (multiple of chunk)
    float *seg_S, *seg_z;              // [BH][nseg+1][D][dv], [BH][nseg+1][D]: prefix at each segment start, total last
    float *seg_dS, *seg_dz;            // [BH][nseg][D][dv], [BH][nseg][D]: suffix after segment end
    float *rowstat;                    // [BH][n][2]: (den_i, dden_i) of the backward pass
    // streaming-form backward on tensor cores
    float *dphi;                       // [BH][n][D] fp32: dLoss/dphi of Q, then of K
    void *phik, *pq2;                  // [BH][n][2D] bf16 phi(k), phi(q)/den, each as (hi | lo)
    // tensor-core work items balanced by valid tiles (non-causal, with lengths): workspace for the split
    // ([kMaxGrid + 1] block starts, [2*BH] runs), and the split in use (null: by count)
    // per-head parameters run one sub-problem per head index h (over the B sequences): head bh of the
    // sub-problem is head bh * hs_mul of the caller's tensors and state (base pointers already offset to
    // head h); hs_mul = 1 otherwise
    int hs_mul;
    int *items_ws;
    const int *split;                  // block b takes items split[b] .. split[b+1]-1
    const int *runs;                   // [2*BH]: first and last block holding an item of head bh
    int padded_zeroed;                 // the outputs' rows past each sequence's length are already zero
    // channel RMS normalisation of the feature map (non-causal; ch_sigma null: off)
    float ch_target;                   // the listing's ch_rms_target
    luna_dtype ch_io;                  // element type of Q, K, dQ, dK
    float *ch_part;                    // [2][kChStatBlocks][L]: per-block sums of phi^2, queries then keys
    double *ch_stat;                   // [8][kMaxL]: per side s, rms, target/(rms+eps), unused; [3][0] = N
    float *ch_sigma;                   // [kMaxL]: s^q_l s^k_l
    double *ch_T;                      // [BH][L]: per-head sums of S' . dS + z' dz over each channel's rows
                                       // (streaming form: [ch_T_rows][L] block sums of phi^ . dLoss/dphi^)
    float *ch_kappa;                   // [2][kMaxL]: factor of y_l in dLoss/dy_l from the scale, per side
    int ch_causal;                     // streaming form: the kernels run on the sqrt(sigma)-scaled table
    int ch_T_rows;                     // rows of ch_T written by the streaming form's chain rule
};

// Row offset of head bh in the caller's tensors (Q, K, V, dO, O, dQ, dK, dV), and its index among the
// caller's per-head state blocks (S, z; the streaming form's segment prefixes).
__host__ __device__ inline size_t head_rows(const AttnArgs &a, int bh) { return (size_t)bh * a.hs_mul * a.n; }
__host__ __device__ inline size_t head_state(const AttnArgs &a, int bh) { return (size_t)bh * a.hs_mul; }

// blocks per side of the channel-statistics kernel and of the scale-term backward pass (fixed counts:
// the sums do not depend on the device)
constexpr int kChStatBlocks = 304;
constexpr int kChKBlocks = 304;

// one step of the streaming form for every (batch, head): state S [D][dv], z [D] (fp32, in place)
struct DecodeArgs {
    int BH, d, dv, M, L, D;
    float eps;
    TableLayout lay;
    const char *table;
    int H;                       // heads per sequence
    int64_t table_stride;        // bytes between heads' tables (per-head parameters), 0: one shared table
    const void *q, *k, *v;
    void *o;
    float *S, *z;
    int64_t S_stride, z_stride;  // elements between consecutive heads
};
cudaError_t launch_decode(const DecodeArgs &a, luna_dtype io, cudaStream_t s);
cudaError_t launch_selftest_wait(int *status, long long limit_ns, cudaStream_t s);

cudaError_t launch_phi_prepare(const luna_phi_params &prm, const TableLayout &lay, void *table, cudaStream_t s);
cudaError_t launch_featmap(const TableLayout &lay, const char *table, const void *X, luna_dtype xt, int64_t rows,
                           float *Phi, cudaStream_t s);
cudaError_t launch_simt_fwd(const AttnArgs &a, luna_dtype io, cudaStream_t s);
cudaError_t launch_simt_stats(const AttnArgs &a, luna_dtype io, cudaStream_t s);
cudaError_t launch_simt_bwd(const AttnArgs &a, luna_dtype io, bool have_stats, cudaStream_t s);
cudaError_t launch_grad_reduce(const AttnArgs &a, int nparts, cudaStream_t s);
cudaError_t launch_causal_fwd(const AttnArgs &a, luna_dtype io, bool write_state, cudaStream_t s);
cudaError_t launch_causal_bwd(const AttnArgs &a, luna_dtype io, bool have_state, cudaStream_t s);
size_t simt_max_smem(const AttnArgs &a);
// attention weights of query rows [row0, row0 + rows) of every head (conversion, stage 1): A (BH, rows, n)
cudaError_t launch_weights(const AttnArgs &a, luna_dtype io, int causal, int row0, int rows, int teacher,
                           int64_t tstride, float *A, cudaStream_t s);
size_t weights_max_smem(const AttnArgs &a);
// channel RMS normalisation: statistics and scales of both sides; S, z rows times sigma (after any key
// statistics); dS, dz rows times sigma and the per-head sums T (between the query- and key-side backward
// kernels); the scale term of the backward (before the parameter-gradient reduction: its partials follow
// the main_parts ones, *nparts is the new count).  Each is a no-op when ch_sigma is null.
cudaError_t launch_chrms_stats(const AttnArgs &a, luna_dtype io, cudaStream_t s);
cudaError_t launch_chrms_scale_state(const AttnArgs &a, cudaStream_t s);
cudaError_t launch_chrms_dstate(const AttnArgs &a, cudaStream_t s);
cudaError_t launch_chrms_backward(const AttnArgs &a, int main_parts, int *nparts, cudaStream_t s);
// streaming form: the table with channel l's coefficients times sqrt(sigma_l) into dst (a.lay.bytes), and
// the reduced histogram's channel l times sqrt(sigma_l) (between the partial sum and the MLP gradients)
cudaError_t launch_chrms_table(const AttnArgs &a, char *dst, cudaStream_t s);
// kappa of both sides from the T rows (the streaming form on tensor cores folds it into its chain rule)
cudaError_t launch_chrms_kappa(const AttnArgs &a, cudaStream_t s);
cudaError_t launch_chrms_hist(const AttnArgs &a, cudaStream_t s);
size_t chrms_max_smem(const AttnArgs &a);
size_t causal_max_smem(const AttnArgs &a);

}  // namespace luna
