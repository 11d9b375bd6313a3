// Streaming (causal) form on CUDA cores (fp32 arithmetic).
//
// The paper names the associative streaming form of kernel attention (abstract,
// Sec. 3.2, Conclusion) without writing it out; it is the prefix recurrence
//     S_i = S_{i-1} + phi(k_i) v_i^T,  z_i = z_{i-1} + phi(k_i),
//     O_i = phi(q_i)^T S_i / (phi(q_i)^T z_i + eps).
// Rows are cut into state segments.  The prefix statistics at every segment
// start come from an exclusive scan of per-segment sums (key-statistics kernel
// in scan mode); inside a segment the rows are processed in sub-chunks of kCs
// rows: a masked intra-chunk term tril(phi(Q) phi(K)^T) V plus the carried
// state, then the state advances by the chunk's phi(K)^T V.
//
// Backward (derived from the same recurrence):
//   dnum_i = do_i / den_i, dden_i = -(do_i . o_i)/den_i
//   dphi(q_i) = S_i dnum_i + z_i dden_i
//   G_j = sum_{i>=j} phi(q_i) dnum_i^T, g_j = sum_{i>=j} phi(q_i) dden_i
//   dv_j = G_j^T phi(k_j),  dphi(k_j) = G_j v_j + g_j
// A forward sweep per segment records (den_i, dden_i) and the segment sums of
// G; a reverse exclusive scan gives G after every segment; then one forward
// sweep produces dQ and one reverse sweep produces dK and dV.
#include <math.h>

#include "luna_prof.cuh"
#include "luna_simt_dev.cuh"

namespace luna {
namespace {
using namespace simt;

constexpr int kCs = 16;  // rows per sub-chunk

struct ChunkBufs {
    float *Q, *K, *V, *dO, *Pq, *Pk, *A, *P, *den, *dden;
};

template <typename IO>
__device__ void load_chunk(const AttnArgs &a, int bh, int t0, int nr, float *sQ, float *sK, float *sV, float *sdO) {
    const size_t r0 = head_rows(a, bh) + t0;
    load_rows(sQ, static_cast<const IO *>(a.Q) + r0 * a.d, nr * a.d);
    load_rows(sK, static_cast<const IO *>(a.K) + r0 * a.d, nr * a.d);
    load_rows(sV, static_cast<const IO *>(a.V) + r0 * a.dv, nr * a.dv);
    if (sdO) load_rows(sdO, static_cast<const IO *>(a.dO) + r0 * a.dv, nr * a.dv);
}

// sA[r][j] = phi(q_r) . phi(k_j) for j <= r (0 above the diagonal)
__device__ void masked_scores(const float *sPq, const float *sPk, int nr, int D, float *sA) {
    for (int e = threadIdx.x; e < nr * kCs; e += blockDim.x) {
        const int r = e / kCs, j = e - r * kCs;
        float acc = 0.0f;
        if (j <= r && j < nr)
            for (int f = 0; f < D; ++f) acc = fmaf(sPq[r * D + f], sPk[j * D + f], acc);
        sA[e] = acc;
    }
}

// state update S += phi(K)^T V, z += sum phi(K) over the chunk rows (fp64, one rounding per chunk: the
// running state is shared by every later row, so its rounding does not average out in the gradients)
__device__ void advance_state(float *S, float *z, const float *sPk, const float *sV, int nr, int D, int dv) {
    for (int e = threadIdx.x; e < D * dv; e += blockDim.x) {
        const int f = e / dv, c = e - f * dv;
        double acc = S[e];
        for (int r = 0; r < nr; ++r) acc = fma((double)sPk[r * D + f], (double)sV[r * dv + c], acc);
        S[e] = (float)acc;
    }
    for (int f = threadIdx.x; f < D; f += blockDim.x) {
        double acc = z[f];
        for (int r = 0; r < nr; ++r) acc += (double)sPk[r * D + f];
        z[f] = (float)acc;
    }
}

// den_r = eps + phi(q_r).z + sum_{j<=r} A[r][j];  O_r = (phi(q_r) S + sum_{j<=r} A[r][j] v_j) / den_r,
// both formed in fp64 and rounded once (the backward's gradients cancel to a small part of their terms
// under the scale invariance of each row, so a row's rounding must stay at half an ulp)
__device__ void chunk_outputs(const AttnArgs &a, const float *S, const float *z, const float *sPq, const float *sA,
                              const float *sV, int nr, float *sden, float *sO) {
    const int D = a.D, dv = a.dv;
    for (int r = threadIdx.x; r < nr; r += blockDim.x) {
        double den = a.eps;
        for (int f = 0; f < D; ++f) den = fma((double)sPq[r * D + f], (double)z[f], den);
        for (int j = 0; j <= r; ++j) den += (double)sA[r * kCs + j];
        sden[r] = (float)den;
    }
    __syncthreads();
    for (int e = threadIdx.x; e < nr * dv; e += blockDim.x) {
        const int r = e / dv, c = e - r * dv;
        float o = 0.0f;
        if (sden[r] != 0.0f) {
            double num = 0.0;
            for (int f = 0; f < D; ++f) num = fma((double)sPq[r * D + f], (double)S[f * dv + c], num);
            for (int j = 0; j <= r; ++j) num = fma((double)sA[r * kCs + j], (double)sV[j * dv + c], num);
            o = (float)(num / (double)sden[r]);
        }
        sO[e] = o;
    }
}

// ---------------------------------------------------------------------------

template <typename IO>
__global__ void __launch_bounds__(kThreads) k_causal_out(AttnArgs a) {
    extern __shared__ __align__(16) float smem[];
    Carve cv{smem};
    const TableLayout &lay = a.lay;
    const int D = a.D, dv = a.dv, d = a.d;
    SmemPhi s = carve_phi(cv, lay);
    float *S = cv.take(D * dv), *z = cv.take(D);
    float *sQ = cv.take(kCs * d), *sK = cv.take(kCs * d), *sV = cv.take(kCs * dv);
    float *sPq = cv.take(kCs * D), *sPk = cv.take(kCs * D), *sA = cv.take(kCs * kCs);
    float *sden = cv.take(kCs), *sO = cv.take(kCs * dv);
    if (!carve_fits(cv, smem)) return;
    const int bh = blockIdx.y, seg = blockIdx.x;
    const int len = head_length(a.lengths, bh / a.H, a.n);
    const int r0 = seg * a.seg_len, rend = min(a.n, r0 + a.seg_len), r1 = min(len, rend);
    IO *O = static_cast<IO *>(a.O) + head_rows(a, bh) * dv;
    for (int e = threadIdx.x + max(r0, len) * dv; e < rend * dv; e += blockDim.x) io_store(O + e, 0.0f);
    if (r0 >= r1) return;
    load_phi(s, lay, a.table);
    const size_t so = head_state(a, bh) * (a.nseg + 1) + seg;
    for (int e = threadIdx.x; e < D * dv; e += blockDim.x) S[e] = a.seg_S[so * D * dv + e];
    for (int e = threadIdx.x; e < D; e += blockDim.x) z[e] = a.seg_z[so * D + e];
    for (int t0 = r0; t0 < r1; t0 += kCs) {
        const int nr = min(kCs, r1 - t0);
        __syncthreads();
        load_chunk<IO>(a, bh, t0, nr, sQ, sK, sV, nullptr);
        __syncthreads();
        phi_tile(lay, s, sQ, nr, sPq, nullptr, nullptr);
        phi_tile(lay, s, sK, nr, sPk, nullptr, nullptr);
        __syncthreads();
        masked_scores(sPq, sPk, nr, D, sA);
        __syncthreads();
        chunk_outputs(a, S, z, sPq, sA, sV, nr, sden, sO);
        __syncthreads();
        for (int e = threadIdx.x; e < nr * dv; e += blockDim.x) io_store(O + (size_t)t0 * dv + e, sO[e]);
        advance_state(S, z, sPk, sV, nr, D, dv);
    }
}

// forward sweep of the backward pass: records (den_i, dden_i), sums G over the segment
template <typename IO>
__global__ void __launch_bounds__(kThreads) k_causal_bwd_seg(AttnArgs a) {
    extern __shared__ __align__(16) float smem[];
    Carve cv{smem};
    const TableLayout &lay = a.lay;
    const int D = a.D, dv = a.dv, d = a.d;
    SmemPhi s = carve_phi(cv, lay);
    float *S = cv.take(D * dv), *z = cv.take(D);
    float *sQ = cv.take(kCs * d), *sK = cv.take(kCs * d), *sV = cv.take(kCs * dv), *sdO = cv.take(kCs * dv);
    float *sPq = cv.take(kCs * D), *sPk = cv.take(kCs * D), *sA = cv.take(kCs * kCs);
    float *sden = cv.take(kCs), *sdden = cv.take(kCs), *sO = cv.take(kCs * dv);
    if (!carve_fits(cv, smem)) return;
    const int bh = blockIdx.y, seg = blockIdx.x;
    const int len = head_length(a.lengths, bh / a.H, a.n);
    const int r0 = seg * a.seg_len, rend = min(a.n, r0 + a.seg_len), r1 = min(len, rend);
    load_phi(s, lay, a.table);
    const size_t so = head_state(a, bh) * (a.nseg + 1) + seg;
    for (int e = threadIdx.x; e < D * dv; e += blockDim.x) S[e] = a.seg_S[so * D * dv + e];
    for (int e = threadIdx.x; e < D; e += blockDim.x) z[e] = a.seg_z[so * D + e];
    const int nc = (dv + 7) / 8, nf = (D + 7) / 8;
    const bool active = threadIdx.x < nf * nc;
    const int tf = active ? threadIdx.x / nc : 0, tc = active ? threadIdx.x % nc : 0;
    const int f0 = tf * 8, c0 = tc * 8;
    double acc[8][8] = {}, zacc[8] = {};
    for (int t0 = r0; t0 < r1; t0 += kCs) {
        const int nr = min(kCs, r1 - t0);
        __syncthreads();
        load_chunk<IO>(a, bh, t0, nr, sQ, sK, sV, sdO);
        __syncthreads();
        phi_tile(lay, s, sQ, nr, sPq, nullptr, nullptr);
        phi_tile(lay, s, sK, nr, sPk, nullptr, nullptr);
        __syncthreads();
        masked_scores(sPq, sPk, nr, D, sA);
        __syncthreads();
        chunk_outputs(a, S, z, sPq, sA, sV, nr, sden, sO);
        __syncthreads();
        for (int r = threadIdx.x; r < nr; r += blockDim.x) {
            double dot = 0.0;  // dden and dphi are formed in fp64 and rounded once: they cancel
            for (int c = 0; c < dv; ++c) dot = fma((double)sdO[r * dv + c], (double)sO[r * dv + c], dot);
            const float dd = (sden[r] != 0.0f) ? (float)(-dot / (double)sden[r]) : 0.0f;
            sdden[r] = dd;
            float *rs = a.rowstat + ((size_t)bh * a.n + t0 + r) * 2;
            rs[0] = sden[r];
            rs[1] = dd;
        }
        __syncthreads();
        for (int e = threadIdx.x; e < nr * dv; e += blockDim.x) {
            const int r = e / dv;
            sO[e] = (sden[r] != 0.0f) ? sdO[e] / sden[r] : 0.0f;  // dnum
        }
        __syncthreads();
        if (active) outer_accumulate(acc, zacc, true, sPq, D, sO, dv, sdden, nr, f0, c0);
        advance_state(S, z, sPk, sV, nr, D, dv);
    }
    __syncthreads();
    const size_t slot = (size_t)bh * a.nseg + seg;
    store_tile(acc, zacc, active, tc, f0, c0, D, dv, a.dS_part + slot * D * dv, a.dz_part + slot * D);
    if (last_arrival(a.counters + a.B * a.H + bh, a.nseg)) {
        exclusive_scan(a.dS_part + (size_t)bh * a.nseg * D * dv, a.nseg, D * dv, a.seg_dS + (size_t)bh * a.nseg * D * dv,
                       true);
        exclusive_scan(a.dz_part + (size_t)bh * a.nseg * D, a.nseg, D, a.seg_dz + (size_t)bh * a.nseg * D, true);
        if (threadIdx.x == 0) a.counters[a.B * a.H + bh] = 0;
    }
}

// dQ: forward sweep.  dphi(q_i) = S_{before chunk} dnum_i + z dden_i + sum_{j<=i in chunk} dP_ij phi(k_j),
// dP_ij = dnum_i . v_j + dden_i
template <typename IO>
__global__ void __launch_bounds__(kThreads) k_causal_dq(AttnArgs a) {
    extern __shared__ __align__(16) float smem[];
    Carve cv{smem};
    const TableLayout &lay = a.lay;
    const int D = a.D, dv = a.dv, d = a.d, M = a.M;
    SmemPhi s = carve_phi(cv, lay);
    float *S = cv.take(D * dv), *z = cv.take(D);
    float *sQ = cv.take(kCs * d), *sK = cv.take(kCs * d), *sV = cv.take(kCs * dv), *sdO = cv.take(kCs * dv);
    float *sPq = cv.take(kCs * D), *sPk = cv.take(kCs * D), *sdPq = cv.take(kCs * D), *sP = cv.take(kCs * kCs);
    float *sden = cv.take(kCs), *sdden = cv.take(kCs);
    float *sU = cv.take(kCs * M);
    int *sJ = reinterpret_cast<int *>(cv.take(kCs * M));
    float *sdU = cv.take(kCs * M);
    if (!carve_fits(cv, smem)) return;
    const int bh = blockIdx.y, seg = blockIdx.x;
    __shared__ double sT[kMaxL];  // channel normalisation: the block's sums of phi . dphi per channel
    if ((int)threadIdx.x < kMaxL) sT[threadIdx.x] = 0.0;
    double *gp = reinterpret_cast<double *>(a.gpart) + ((size_t)bh * a.nseg + seg) * a.gsize;
    double *shist = gp + M * d + M;  // the block's fp64 histogram, accumulated in place by L2 atomics
    const int len = head_length(a.lengths, bh / a.H, a.n);
    const int r0 = seg * a.seg_len, rend = min(a.n, r0 + a.seg_len), r1 = min(len, rend);
    IO *dQ = static_cast<IO *>(a.dQ) + head_rows(a, bh) * d;
    for (int e = threadIdx.x + max(r0, len) * d; e < rend * d; e += blockDim.x) io_store(dQ + e, 0.0f);
    load_phi(s, lay, a.table);
    const size_t so = head_state(a, bh) * (a.nseg + 1) + seg;
    for (int e = threadIdx.x; e < D * dv; e += blockDim.x) S[e] = a.seg_S[so * D * dv + e];
    for (int e = threadIdx.x; e < D; e += blockDim.x) z[e] = a.seg_z[so * D + e];
    for (int e = threadIdx.x; e < mlp_words(lay) + var_words(lay); e += blockDim.x) shist[e] = 0.0;
    GradAcc g = {};
    for (int t0 = r0; t0 < r1; t0 += kCs) {
        const int nr = min(kCs, r1 - t0);
        __syncthreads();
        load_chunk<IO>(a, bh, t0, nr, sQ, sK, sV, sdO);
        for (int r = threadIdx.x; r < nr; r += blockDim.x) {
            const float *rs = a.rowstat + ((size_t)bh * a.n + t0 + r) * 2;
            sden[r] = rs[0];
            sdden[r] = rs[1];
        }
        __syncthreads();
        phi_tile(lay, s, sQ, nr, sPq, sU, sJ);
        phi_tile(lay, s, sK, nr, sPk, nullptr, nullptr);
        for (int e = threadIdx.x; e < nr * dv; e += blockDim.x) {
            const int r = e / dv;
            sdO[e] = (sden[r] != 0.0f) ? sdO[e] / sden[r] : 0.0f;  // dnum in place
        }
        __syncthreads();
        for (int e = threadIdx.x; e < nr * kCs; e += blockDim.x) {
            const int r = e / kCs, j = e - r * kCs;
            double acc = 0.0;
            if (j <= r && j < nr) {
                for (int c = 0; c < dv; ++c) acc = fma((double)sdO[r * dv + c], (double)sV[j * dv + c], acc);
                acc += (double)sdden[r];
            }
            sP[e] = (float)acc;
        }
        __syncthreads();
        for (int e = threadIdx.x; e < nr * D; e += blockDim.x) {
            const int r = e / D, f = e - r * D;
            double acc = (double)z[f] * (double)sdden[r];
            for (int c = 0; c < dv; ++c) acc = fma((double)S[f * dv + c], (double)sdO[r * dv + c], acc);
            for (int j = 0; j <= r; ++j) acc = fma((double)sP[r * kCs + j], (double)sPk[j * D + f], acc);
            sdPq[e] = (float)acc;
            if (a.ch_T) atomicAdd(sT + f % a.L, (double)sPq[e] * acc);
        }
        __syncthreads();
        advance_state(S, z, sPk, sV, nr, D, dv);
        phi_backward_tile(lay, s, sQ, nr, sPq, sdPq, sU, sJ, sdU, shist, shist + mlp_words(lay), g);
        store_dx(lay, s, sdU, nr, dQ + (size_t)t0 * d);
    }
    __syncthreads();
    store_grad_partial(lay, g, gp);
    if (a.ch_T && (int)threadIdx.x < a.L) a.ch_T[((size_t)bh * a.nseg + seg) * a.L + threadIdx.x] = sT[threadIdx.x];
}

// dK, dV: reverse sweep with the suffix state G (after the current chunk).
//   dv_j = G^T phi(k_j) + sum_{i>=j in chunk} A_ij dnum_i
//   dphi(k_j) = G v_j + g + sum_{i>=j in chunk} dP_ij phi(q_i)
template <typename IO>
__global__ void __launch_bounds__(kThreads) k_causal_dkv(AttnArgs a) {
    extern __shared__ __align__(16) float smem[];
    Carve cv{smem};
    const TableLayout &lay = a.lay;
    const int D = a.D, dv = a.dv, d = a.d, M = a.M;
    SmemPhi s = carve_phi(cv, lay);
    float *G = cv.take(D * dv), *gz = cv.take(D);
    float *sQ = cv.take(kCs * d), *sK = cv.take(kCs * d), *sV = cv.take(kCs * dv), *sdO = cv.take(kCs * dv);
    float *sPq = cv.take(kCs * D), *sPk = cv.take(kCs * D), *sdPk = cv.take(kCs * D);
    float *sA = cv.take(kCs * kCs), *sP = cv.take(kCs * kCs);
    float *sden = cv.take(kCs), *sdden = cv.take(kCs);
    float *sU = cv.take(kCs * M);
    int *sJ = reinterpret_cast<int *>(cv.take(kCs * M));
    float *sdU = cv.take(kCs * M);
    if (!carve_fits(cv, smem)) return;
    const int bh = blockIdx.y, seg = blockIdx.x;
    double *gp = reinterpret_cast<double *>(a.gpart) + ((size_t)a.B * a.H * a.nseg + (size_t)bh * a.nseg + seg) * a.gsize;
    double *shist = gp + M * d + M;  // the block's fp64 histogram, accumulated in place by L2 atomics
    const int len = head_length(a.lengths, bh / a.H, a.n);
    const int r0 = seg * a.seg_len, rend = min(a.n, r0 + a.seg_len), r1 = min(len, rend);
    IO *dK = static_cast<IO *>(a.dK) + head_rows(a, bh) * d;
    IO *dV = static_cast<IO *>(a.dV) + head_rows(a, bh) * dv;
    for (int e = threadIdx.x + max(r0, len) * d; e < rend * d; e += blockDim.x) io_store(dK + e, 0.0f);
    for (int e = threadIdx.x + max(r0, len) * dv; e < rend * dv; e += blockDim.x) io_store(dV + e, 0.0f);
    load_phi(s, lay, a.table);
    const size_t so = (size_t)bh * a.nseg + seg;
    for (int e = threadIdx.x; e < D * dv; e += blockDim.x) G[e] = a.seg_dS[so * D * dv + e];
    for (int e = threadIdx.x; e < D; e += blockDim.x) gz[e] = a.seg_dz[so * D + e];
    for (int e = threadIdx.x; e < mlp_words(lay) + var_words(lay); e += blockDim.x) shist[e] = 0.0;
    GradAcc g = {};
    if (r1 > r0) {
        for (int t0 = r0 + ((r1 - 1 - r0) / kCs) * kCs; t0 >= r0; t0 -= kCs) {
            const int nr = min(kCs, r1 - t0);
            __syncthreads();
            load_chunk<IO>(a, bh, t0, nr, sQ, sK, sV, sdO);
            for (int r = threadIdx.x; r < nr; r += blockDim.x) {
                const float *rs = a.rowstat + ((size_t)bh * a.n + t0 + r) * 2;
                sden[r] = rs[0];
                sdden[r] = rs[1];
            }
            __syncthreads();
            phi_tile(lay, s, sQ, nr, sPq, nullptr, nullptr);
            phi_tile(lay, s, sK, nr, sPk, sU, sJ);
            for (int e = threadIdx.x; e < nr * dv; e += blockDim.x) {
                const int r = e / dv;
                sdO[e] = (sden[r] != 0.0f) ? sdO[e] / sden[r] : 0.0f;  // dnum in place
            }
            __syncthreads();
            masked_scores(sPq, sPk, nr, D, sA);
            for (int e = threadIdx.x; e < nr * kCs; e += blockDim.x) {
                const int r = e / kCs, j = e - r * kCs;
                double acc = 0.0;
                if (j <= r && j < nr) {
                    for (int c = 0; c < dv; ++c) acc = fma((double)sdO[r * dv + c], (double)sV[j * dv + c], acc);
                    acc += (double)sdden[r];
                }
                sP[e] = (float)acc;
            }
            __syncthreads();
            for (int e = threadIdx.x; e < nr * dv; e += blockDim.x) {
                const int j = e / dv, c = e - j * dv;
                float acc = 0.0f;
                for (int f = 0; f < D; ++f) acc = fmaf(G[f * dv + c], sPk[j * D + f], acc);
                for (int r = j; r < nr; ++r) acc = fmaf(sA[r * kCs + j], sdO[r * dv + c], acc);
                io_store(dV + (size_t)t0 * dv + e, acc);
            }
            for (int e = threadIdx.x; e < nr * D; e += blockDim.x) {
                const int j = e / D, f = e - j * D;
                double acc = gz[f];
                for (int c = 0; c < dv; ++c) acc = fma((double)G[f * dv + c], (double)sV[j * dv + c], acc);
                for (int r = j; r < nr; ++r) acc = fma((double)sP[r * kCs + j], (double)sPq[r * D + f], acc);
                sdPk[e] = (float)acc;
            }
            __syncthreads();
            // G += phi(Q_chunk)^T dnum, g += phi(Q_chunk)^T dden
            for (int e = threadIdx.x; e < D * dv; e += blockDim.x) {
                const int f = e / dv, c = e - f * dv;
                double acc = G[e];
                for (int r = 0; r < nr; ++r) acc = fma((double)sPq[r * D + f], (double)sdO[r * dv + c], acc);
                G[e] = (float)acc;
            }
            for (int f = threadIdx.x; f < D; f += blockDim.x) {
                double acc = gz[f];
                for (int r = 0; r < nr; ++r) acc = fma((double)sPq[r * D + f], (double)sdden[r], acc);
                gz[f] = (float)acc;
            }
            phi_backward_tile(lay, s, sK, nr, sPk, sdPk, sU, sJ, sdU, shist, shist + mlp_words(lay), g);
            store_dx(lay, s, sdU, nr, dK + (size_t)t0 * d);
        }
    }
    __syncthreads();
    store_grad_partial(lay, g, gp);
}

// ---------------------------------------------------------------------------

size_t smem_out(const AttnArgs &a) {
    HostCarve cv; carve_phi_host(cv, a.lay);
    cv.take(a.D * a.dv); cv.take(a.D); cv.take(kCs * a.d); cv.take(kCs * a.d); cv.take(kCs * a.dv);
    cv.take(kCs * a.D); cv.take(kCs * a.D); cv.take(kCs * kCs); cv.take(kCs); cv.take(kCs * a.dv);
    return cv.bytes();
}
size_t smem_bwd_seg(const AttnArgs &a) {
    return smem_out(a) + 4 * (size_t)(r4(kCs * a.dv) + r4(kCs));
}
size_t smem_dq(const AttnArgs &a) {
    HostCarve cv; carve_phi_host(cv, a.lay);
    cv.take(a.D * a.dv); cv.take(a.D); cv.take(kCs * a.d); cv.take(kCs * a.d); cv.take(kCs * a.dv);
    cv.take(kCs * a.dv); cv.take(kCs * a.D); cv.take(kCs * a.D); cv.take(kCs * a.D); cv.take(kCs * kCs);
    cv.take(kCs); cv.take(kCs); cv.take(kCs * a.M); cv.take(kCs * a.M); cv.take(kCs * a.M);
    return cv.bytes();
}
size_t smem_dkv(const AttnArgs &a) { return smem_dq(a) + 4 * (size_t)r4(kCs * kCs); }

template <typename IO>
cudaError_t seg_stats(const AttnArgs &a, cudaStream_t s) {
    AttnArgs b = a;
    b.nsplit = a.nseg;
    b.rows_per_split = a.seg_len;
    return launch_simt_stats(b, IOType<IO>::code, s);
}

template <typename IO>
cudaError_t causal_fwd_impl(const AttnArgs &a, cudaStream_t s) {
    cudaError_t e = seg_stats<IO>(a, s);
    if (e != cudaSuccess) return e;
    const size_t sm = smem_out(a);
    if ((e = set_smem(k_causal_out<IO>, sm)) != cudaSuccess) return e;
    LUNA_LAUNCH("causal_out", k_causal_out<IO>, dim3(a.nseg, a.B * a.H), kThreads, sm, s, a);
    return cudaGetLastError();
}

template <typename IO>
cudaError_t causal_bwd_impl(const AttnArgs &a0, bool have_state, cudaStream_t s) {
    AttnArgs a = a0;
    a.gpart64 = 1;  // the generic kernels write fp64 parameter-gradient partials
    cudaError_t e;
    if (!have_state && (e = seg_stats<IO>(a, s)) != cudaSuccess) return e;
    const dim3 grid(a.nseg, a.B * a.H);
    size_t sm = smem_bwd_seg(a);
    if ((e = set_smem(k_causal_bwd_seg<IO>, sm)) != cudaSuccess) return e;
    LUNA_LAUNCH("causal_bwd_seg", k_causal_bwd_seg<IO>, grid, kThreads, sm, s, a);
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
    sm = smem_dq(a);
    if ((e = set_smem(k_causal_dq<IO>, sm)) != cudaSuccess) return e;
    LUNA_LAUNCH("causal_dq", k_causal_dq<IO>, grid, kThreads, sm, s, a);
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
    sm = smem_dkv(a);
    if ((e = set_smem(k_causal_dkv<IO>, sm)) != cudaSuccess) return e;
    LUNA_LAUNCH("causal_dkv", k_causal_dkv<IO>, grid, kThreads, sm, s, a);
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
    int nparts = 2 * a.B * a.H * a.nseg;
    if (a.ch_sigma) {  // the scale term of the channel normalisation (kappa from the queries' T rows)
        a.ch_T_rows = a.B * a.H * a.nseg;
        if ((e = launch_chrms_backward(a, nparts, &nparts, s)) != cudaSuccess) return e;
    }
    return launch_grad_reduce(a, nparts, s);
}

}  // namespace

size_t causal_max_smem(const AttnArgs &a) {
    size_t m = smem_out(a);
    if (smem_bwd_seg(a) > m) m = smem_bwd_seg(a);
    if (smem_dq(a) > m) m = smem_dq(a);
    if (smem_dkv(a) > m) m = smem_dkv(a);
    return m;
}

cudaError_t launch_causal_fwd(const AttnArgs &a, luna_dtype io, bool, cudaStream_t s) {
    return io == LUNA_F32 ? causal_fwd_impl<float>(a, s) : causal_fwd_impl<__nv_bfloat16>(a, s);
}

cudaError_t launch_causal_bwd(const AttnArgs &a, luna_dtype io, bool have_state, cudaStream_t s) {
    return io == LUNA_F32 ? causal_bwd_impl<float>(a, have_state, s) : causal_bwd_impl<__nv_bfloat16>(a, have_state, s);
}

}  // namespace luna
