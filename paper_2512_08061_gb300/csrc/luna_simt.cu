// Generic CUDA-core kernels of the LUNA attention path (fp32 arithmetic).
//
// They serve the fp32 I/O path (the parity bar there is 1e-4 relative, which
// rules out bf16 tensor-core operands) and every shape the tensor-core path
// does not specialise.  One thread block owns a (head, row range); all
// statistics are fp32 and every cross-block reduction is performed in a fixed
// order by the last block to arrive, so results are reproducible run to run
// except for the order of shared-memory atomic adds in the gradient
// histograms of the channel-MLP parameters.
#include <math.h>

#include "luna_prof.cuh"
#include "luna_simt_dev.cuh"

namespace luna {
namespace {
using namespace simt;

// ---------------------------------------------------------------------------
// feature map alone

template <typename IO>
__global__ void __launch_bounds__(kThreads) k_featmap(TableLayout lay, const char *table, const IO *X, int64_t rows,
                                                      float *Phi) {
    extern __shared__ __align__(16) float smem[];
    __shared__ __align__(16) float sS[kEytzinger];  // the interval search block (the tensor-core kernels' lookup)
    Carve cv{smem};
    SmemPhi s = carve_phi(cv, lay);
    if (!carve_fits(cv, smem)) return;
    load_phi(s, lay, table);
    for (int e = threadIdx.x; e < kEytzinger; e += blockDim.x) sS[e] = reinterpret_cast<const float *>(table + lay.off_Te)[e];
    __syncthreads();
    const unsigned short *sB = reinterpret_cast<const unsigned short *>(sS + kSearchT);
    const int M = lay.M, L = lay.L, d = lay.d, D = lay.D;
    for (int64_t e = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; e < rows * M; e += (int64_t)gridDim.x * blockDim.x) {
        const int64_t r = e / M;
        const int i = (int)(e - r * M);
        const IO *x = X + r * d;
        const float *w = s.W + i * d;
        float u = s.b[i];
        for (int c = 0; c < d; ++c) u = fmaf(w[c], io_load(x + c), u);
        const int j = interval_bucketed(sS, sB, u);
        const float *ab = s.AB + j * ab_stride(lay);
        float *out = Phi + r * D + i * L;
        for (int l = 0; l < L; ++l) {
            const float2 p = ab_pair(ab, l);
            out[l] = fmaxf(fmaf(p.x, u, p.y), channel_floor(lay));
        }
    }
}

// The feature map of the variants (a non-ReLU activation, the envelope gate, Bank+Coef): blocks walk tiles of
// kPhiRows rows through the generic tile helper.
template <typename IO>
__global__ void __launch_bounds__(kThreads) k_featmap_var(TableLayout lay, const char *table, const IO *X,
                                                          int64_t rows, float *Phi) {
    extern __shared__ __align__(16) float smem[];
    Carve cv{smem};
    SmemPhi s = carve_phi(cv, lay);
    float *sX = cv.take(kPhiRows * lay.d);
    float *sPhi = cv.take(kPhiRows * lay.D);
    if (!carve_fits(cv, smem)) return;
    load_phi(s, lay, table);
    for (int64_t t0 = (int64_t)blockIdx.x * kPhiRows; t0 < rows; t0 += (int64_t)gridDim.x * kPhiRows) {
        const int nr = (int)(rows - t0 < kPhiRows ? rows - t0 : kPhiRows);
        __syncthreads();
        load_rows(sX, X + t0 * lay.d, nr * lay.d);
        __syncthreads();
        phi_tile(lay, s, sX, nr, sPhi, nullptr, nullptr);
        __syncthreads();
        for (int e = threadIdx.x; e < nr * lay.D; e += blockDim.x) Phi[t0 * lay.D + e] = sPhi[e];
    }
}

// ---------------------------------------------------------------------------
// key statistics S = sum_j phi(k_j) v_j^T, z = sum_j phi(k_j)   (Sec. 4: S_KV, S_K1)

template <typename IO>
__global__ void __launch_bounds__(kThreads) k_keystats(AttnArgs a) {
    extern __shared__ __align__(16) float smem[];
    Carve cv{smem};
    const TableLayout &lay = a.lay;
    SmemPhi s = carve_phi(cv, lay);
    float *sK = cv.take(kTileK * a.d);
    float *sV = cv.take(kTileK * a.dv);
    float *sPhi = cv.take(kTileK * a.D);
    if (!carve_fits(cv, smem)) return;
    load_phi(s, lay, a.table);

    const int bh = blockIdx.y, split = blockIdx.x;
    const int len = head_length(a.lengths, bh / a.H, a.n);
    const int r0 = split * a.rows_per_split;
    const int r1 = min(len, r0 + a.rows_per_split);
    const IO *K = static_cast<const IO *>(a.K) + head_rows(a, bh) * a.d;
    const IO *V = static_cast<const IO *>(a.V) + head_rows(a, bh) * a.dv;

    const int nc = (a.dv + 7) / 8, nf = (a.D + 7) / 8;
    const bool active = threadIdx.x < nf * nc;
    const int tf = active ? threadIdx.x / nc : 0, tc = active ? threadIdx.x % nc : 0;
    const int f0 = tf * 8, c0 = tc * 8;
    double acc[8][8] = {}, zacc[8] = {};
    for (int t0 = r0; t0 < r1; t0 += kTileK) {
        const int nr = min(kTileK, r1 - t0);
        __syncthreads();
        load_rows(sK, K + (size_t)t0 * a.d, nr * a.d);
        load_rows(sV, V + (size_t)t0 * a.dv, nr * a.dv);
        __syncthreads();
        phi_tile(lay, s, sK, nr, sPhi, nullptr, nullptr);
        __syncthreads();
        if (active) outer_accumulate(acc, zacc, true, sPhi, a.D, sV, a.dv, nullptr, nr, f0, c0);
    }
    const size_t slot = (size_t)bh * a.nsplit + split;
    store_tile(acc, zacc, active, tc, f0, c0, a.D, a.dv, a.S_part + slot * a.D * a.dv, a.z_part + slot * a.D);
    if (last_arrival(a.counters + bh, a.nsplit)) {
        if (a.seg_S) {  // causal: exclusive prefix at every segment start, total in slot nsplit
            exclusive_scan(a.S_part + (size_t)bh * a.nsplit * a.D * a.dv, a.nsplit, a.D * a.dv,
                           a.seg_S + head_state(a, bh) * (a.nsplit + 1) * a.D * a.dv, false);
            exclusive_scan(a.z_part + (size_t)bh * a.nsplit * a.D, a.nsplit, a.D,
                           a.seg_z + head_state(a, bh) * (a.nsplit + 1) * a.D, false);
        } else {
            ordered_sum(a.S_part + (size_t)bh * a.nsplit * a.D * a.dv, a.nsplit, a.D * a.dv,
                        a.S_fin + head_state(a, bh) * a.D * a.dv);
            ordered_sum(a.z_part + (size_t)bh * a.nsplit * a.D, a.nsplit, a.D, a.z_fin + head_state(a, bh) * a.D);
        }
        if (threadIdx.x == 0) a.counters[bh] = 0;
    }
}

// ---------------------------------------------------------------------------
// query side: O_i = phi(q_i)^T S / (phi(q_i)^T z + eps)   (Eq. kernel-attn)

template <typename IO>
__global__ void __launch_bounds__(kThreads) k_query(AttnArgs a) {
    extern __shared__ __align__(16) float smem[];
    const int bh = blockIdx.y;
    const int q0 = blockIdx.x * kTileQ;
    const int len = head_length(a.lengths, bh / a.H, a.n);
    IO *O = static_cast<IO *>(a.O) + head_rows(a, bh) * a.dv;
    const int nrows = min(kTileQ, a.n - q0);
    if (q0 >= len) {  // padded rows only
        for (int e = threadIdx.x; e < nrows * a.dv; e += blockDim.x) io_store(O + (size_t)q0 * a.dv + e, 0.0f);
        return;
    }
    Carve cv{smem};
    const TableLayout &lay = a.lay;
    SmemPhi s = carve_phi(cv, lay);
    float *sS = cv.take(a.D * a.dv);
    float *sz = cv.take(a.D);
    float *sQ = cv.take(kTileQ * a.d);
    float *sPhi = cv.take(kTileQ * a.D);
    float *sden = cv.take(kTileQ);
    if (!carve_fits(cv, smem)) return;
    load_phi(s, lay, a.table);
    for (int e = threadIdx.x; e < a.D * a.dv; e += blockDim.x) sS[e] = a.S_fin[head_state(a, bh) * a.D * a.dv + e];
    for (int e = threadIdx.x; e < a.D; e += blockDim.x) sz[e] = a.z_fin[head_state(a, bh) * a.D + e];
    const int nr = min(nrows, len - q0);
    load_rows(sQ, static_cast<const IO *>(a.Q) + (head_rows(a, bh) + q0) * a.d, nr * a.d);
    __syncthreads();
    phi_tile(lay, s, sQ, nr, sPhi, nullptr, nullptr);
    __syncthreads();
    for (int r = threadIdx.x; r < nr; r += blockDim.x) {
        float den = a.eps;
        for (int f = 0; f < a.D; ++f) den = fmaf(sPhi[r * a.D + f], sz[f], den);
        sden[r] = den;
    }
    __syncthreads();
    for (int e = threadIdx.x; e < nrows * a.dv; e += blockDim.x) {
        const int r = e / a.dv, c = e - r * a.dv;
        float o = 0.0f;
        if (r < nr && sden[r] != 0.0f) {
            float num = 0.0f;
            for (int f = 0; f < a.D; ++f) num = fmaf(sPhi[r * a.D + f], sS[f * a.dv + c], num);
            o = num / sden[r];
        }
        io_store(O + (size_t)q0 * a.dv + e, o);
    }
}

// query side of the backward pass (non-causal):
//   dnum_i = do_i / den_i,  dden_i = -(do_i . o_i) / den_i
//   dphi(q_i) = S dnum_i + z dden_i,  dS += phi(q_i) dnum_i^T,  dz += phi(q_i) dden_i
template <typename IO>
__global__ void __launch_bounds__(kThreads) k_bwd_query(AttnArgs a) {
    extern __shared__ __align__(16) float smem[];
    Carve cv{smem};
    const TableLayout &lay = a.lay;
    const int D = a.D, dv = a.dv, d = a.d, M = a.M;
    SmemPhi s = carve_phi(cv, lay);
    float *sS = cv.take(D * dv);
    float *sz = cv.take(D);
    float *sQ = cv.take(kTileB * d);
    float *sdO = cv.take(kTileB * dv);
    float *sPhi = cv.take(kTileB * D);
    float *sdPhi = cv.take(kTileB * D);
    float *sdnum = cv.take(kTileB * dv);
    float *sden = cv.take(kTileB);
    float *sdden = cv.take(kTileB);
    float *sU = cv.take(kTileB * M);
    int *sJ = reinterpret_cast<int *>(cv.take(kTileB * M));
    float *sdU = cv.take(kTileB * M);
    if (!carve_fits(cv, smem)) return;
    load_phi(s, lay, a.table);
    const int bh = blockIdx.y, split = blockIdx.x;
    const size_t slot = (size_t)bh * a.nsplit_b + split;
    double *gp = reinterpret_cast<double *>(a.gpart) + slot * a.gsize;
    double *shist = gp + M * d + M;  // the block's fp64 histogram, accumulated in place by L2 atomics
    for (int e = threadIdx.x; e < D * dv; e += blockDim.x) sS[e] = a.S_fin[head_state(a, bh) * D * dv + e];
    for (int e = threadIdx.x; e < D; e += blockDim.x) sz[e] = a.z_fin[head_state(a, bh) * D + e];
    for (int e = threadIdx.x; e < mlp_words(lay) + var_words(lay); e += blockDim.x) shist[e] = 0.0;

    const int len = head_length(a.lengths, bh / a.H, a.n);
    const int r0 = split * a.rows_per_split_b;
    const int rend = min(a.n, r0 + a.rows_per_split_b);
    const int r1 = min(len, rend);
    const IO *Q = static_cast<const IO *>(a.Q) + head_rows(a, bh) * d;
    const IO *dO = static_cast<const IO *>(a.dO) + head_rows(a, bh) * dv;
    IO *dQ = static_cast<IO *>(a.dQ) + head_rows(a, bh) * d;
    // padded rows of this range receive zero gradients
    for (int e = threadIdx.x + max(r0, len) * d; e < rend * d; e += blockDim.x) io_store(dQ + e, 0.0f);

    const int nc = (dv + 7) / 8, nf = (D + 7) / 8;
    const bool active = threadIdx.x < nf * nc;
    const int tf = active ? threadIdx.x / nc : 0, tc = active ? threadIdx.x % nc : 0;
    const int f0 = tf * 8, c0 = tc * 8;
    double acc[8][8] = {}, zacc[8] = {};
    GradAcc g = {};
    for (int t0 = r0; t0 < r1; t0 += kTileB) {
        const int nr = min(kTileB, r1 - t0);
        __syncthreads();
        load_rows(sQ, Q + (size_t)t0 * d, nr * d);
        load_rows(sdO, dO + (size_t)t0 * dv, nr * dv);
        __syncthreads();
        phi_tile(lay, s, sQ, nr, sPhi, sU, sJ);
        __syncthreads();
        // den and o_i are formed in fp64 and rounded once: the gradients below cancel to a small part of
        // their terms (the loss barely changes under a common scale of phi(q_i)), so each row's rounding
        // must stay at half an ulp
        for (int r = threadIdx.x; r < nr; r += blockDim.x) {
            double den = a.eps;
            for (int f = 0; f < D; ++f) den = fma((double)sPhi[r * D + f], (double)sz[f], den);
            sden[r] = (float)den;
        }
        __syncthreads();
        for (int e = threadIdx.x; e < nr * dv; e += blockDim.x) {  // o_i into sdnum for now
            const int r = e / dv, c = e - r * dv;
            float o = 0.0f;
            if (sden[r] != 0.0f) {
                double num = 0.0;
                for (int f = 0; f < D; ++f) num = fma((double)sPhi[r * D + f], (double)sS[f * dv + c], num);
                o = (float)(num / (double)sden[r]);
            }
            sdnum[e] = o;
        }
        __syncthreads();
        for (int r = threadIdx.x; r < nr; r += blockDim.x) {
            double dot = 0.0;  // dden and dphi are formed in fp64 and rounded once: they cancel
            for (int c = 0; c < dv; ++c) dot = fma((double)sdO[r * dv + c], (double)sdnum[r * dv + c], dot);
            sdden[r] = (sden[r] != 0.0f) ? (float)(-dot / (double)sden[r]) : 0.0f;
        }
        __syncthreads();
        for (int e = threadIdx.x; e < nr * dv; e += blockDim.x) {
            const int r = e / dv;
            sdnum[e] = (sden[r] != 0.0f) ? (float)((double)sdO[e] / (double)sden[r]) : 0.0f;
        }
        __syncthreads();
        for (int e = threadIdx.x; e < nr * D; e += blockDim.x) {
            const int r = e / D, f = e - r * D;
            double acc2 = (double)sz[f] * (double)sdden[r];
            for (int c = 0; c < dv; ++c) acc2 = fma((double)sS[f * dv + c], (double)sdnum[r * dv + c], acc2);
            sdPhi[e] = (float)acc2;
        }
        __syncthreads();
        if (active) outer_accumulate(acc, zacc, true, sPhi, D, sdnum, dv, sdden, nr, f0, c0);
        phi_backward_tile(lay, s, sQ, nr, sPhi, sdPhi, sU, sJ, sdU, shist, shist + mlp_words(lay), g);
        store_dx(lay, s, sdU, nr, dQ + (size_t)t0 * d);
    }
    __syncthreads();
    store_tile(acc, zacc, active, tc, f0, c0, D, dv, a.dS_part + slot * D * dv, a.dz_part + slot * D);
    store_grad_partial(lay, g, gp);
    if (last_arrival(a.counters + a.B * a.H + bh, a.nsplit_b)) {
        ordered_sum(a.dS_part + (size_t)bh * a.nsplit_b * D * dv, a.nsplit_b, D * dv, a.dS_fin + (size_t)bh * D * dv);
        ordered_sum(a.dz_part + (size_t)bh * a.nsplit_b * D, a.nsplit_b, D, a.dz_fin + (size_t)bh * D);
        if (threadIdx.x == 0) a.counters[a.B * a.H + bh] = 0;
    }
}

// key side of the backward pass (non-causal):
//   dv_j = dS^T phi(k_j),  dphi(k_j) = dS v_j + dz
template <typename IO>
__global__ void __launch_bounds__(kThreads) k_bwd_key(AttnArgs a) {
    extern __shared__ __align__(16) float smem[];
    Carve cv{smem};
    const TableLayout &lay = a.lay;
    const int D = a.D, dv = a.dv, d = a.d, M = a.M;
    SmemPhi s = carve_phi(cv, lay);
    float *sdS = cv.take(D * dv);
    float *sdz = cv.take(D);
    float *sK = cv.take(kTileB * d);
    float *sV = cv.take(kTileB * dv);
    float *sPhi = cv.take(kTileB * D);
    float *sdPhi = cv.take(kTileB * D);
    float *sU = cv.take(kTileB * M);
    int *sJ = reinterpret_cast<int *>(cv.take(kTileB * M));
    float *sdU = cv.take(kTileB * M);
    if (!carve_fits(cv, smem)) return;
    load_phi(s, lay, a.table);
    const int bh = blockIdx.y, split = blockIdx.x;
    const size_t slot = (size_t)a.B * a.H * a.nsplit_b + (size_t)bh * a.nsplit_b + split;
    double *gp = reinterpret_cast<double *>(a.gpart) + slot * a.gsize;
    double *shist = gp + M * d + M;  // the block's fp64 histogram, accumulated in place by L2 atomics
    for (int e = threadIdx.x; e < D * dv; e += blockDim.x) sdS[e] = a.dS_fin[(size_t)bh * D * dv + e];
    for (int e = threadIdx.x; e < D; e += blockDim.x) sdz[e] = a.dz_fin[(size_t)bh * D + e];
    for (int e = threadIdx.x; e < mlp_words(lay) + var_words(lay); e += blockDim.x) shist[e] = 0.0;

    const int len = head_length(a.lengths, bh / a.H, a.n);
    const int r0 = split * a.rows_per_split_b;
    const int rend = min(a.n, r0 + a.rows_per_split_b);
    const int r1 = min(len, rend);
    const IO *K = static_cast<const IO *>(a.K) + head_rows(a, bh) * d;
    const IO *V = static_cast<const IO *>(a.V) + head_rows(a, bh) * dv;
    IO *dK = static_cast<IO *>(a.dK) + head_rows(a, bh) * d;
    IO *dV = static_cast<IO *>(a.dV) + head_rows(a, bh) * dv;
    for (int e = threadIdx.x + max(r0, len) * d; e < rend * d; e += blockDim.x) io_store(dK + e, 0.0f);
    for (int e = threadIdx.x + max(r0, len) * dv; e < rend * dv; e += blockDim.x) io_store(dV + e, 0.0f);

    GradAcc g = {};
    for (int t0 = r0; t0 < r1; t0 += kTileB) {
        const int nr = min(kTileB, r1 - t0);
        __syncthreads();
        load_rows(sK, K + (size_t)t0 * d, nr * d);
        load_rows(sV, V + (size_t)t0 * dv, nr * dv);
        __syncthreads();
        phi_tile(lay, s, sK, nr, sPhi, sU, sJ);
        __syncthreads();
        for (int e = threadIdx.x; e < nr * dv; e += blockDim.x) {
            const int r = e / dv, c = e - r * dv;
            float acc2 = 0.0f;
            for (int f = 0; f < D; ++f) acc2 = fmaf(sPhi[r * D + f], sdS[f * dv + c], acc2);
            io_store(dV + (size_t)t0 * dv + e, acc2);
        }
        for (int e = threadIdx.x; e < nr * D; e += blockDim.x) {
            const int r = e / D, f = e - r * D;
            double acc2 = sdz[f];
            for (int c = 0; c < dv; ++c) acc2 = fma((double)sdS[f * dv + c], (double)sV[r * dv + c], acc2);
            sdPhi[e] = (float)acc2;
        }
        __syncthreads();
        phi_backward_tile(lay, s, sK, nr, sPhi, sdPhi, sU, sJ, sdU, shist, shist + mlp_words(lay), g);
        store_dx(lay, s, sdU, nr, dK + (size_t)t0 * d);
    }
    __syncthreads();
    store_grad_partial(lay, g, gp);
}

// ---------------------------------------------------------------------------
// parameter gradients: ordered sum of the per-block partials, then the
// channel-MLP gradients from the interval histogram.
//   With g = dLoss/dPhi on active outputs, m0[j][l] = sum g, m1[j][l] = sum g*u
//   over samples falling in interval j; for hidden unit (l,k) active on the
//   intervals A_k:  G0 = sum_{j in A_k} m0, G1 = sum_{j in A_k} m1 and
//     dw2 = (w1 G1 + b1 G0)/sqrt(M), dw1 = w2 G1/sqrt(M), db1 = w2 G0/sqrt(M),
//     db2 = sum_j m0 / sqrt(M).

// Compensated (Neumaier) fp32 summation: s + c carries the running sum with about twice fp32's
// precision (fp64 arithmetic runs at a small fraction of the fp32 rate on this part).
struct CompSum {
    float s = 0.0f, c = 0.0f;
    __device__ __forceinline__ void add(float x) {
        const float t = s + x;
        c += fabsf(s) >= fabsf(x) ? (s - t) + x : (x - t) + s;
        s = t;
    }
};

// Sum of the per-block parameter-gradient partials, in the fixed order p = 0..nparts-1
// per element: 64 elements per block, each summed by 8 threads over consecutive
// eighths of the partials (8 loads in flight; fp32 partials in compensated fp32,
// fp64 partials in fp64), then the eight parts combined in order in fp64.
constexpr int kSumElems = 64, kSumSplit = 8;
template <typename P>
__global__ void __launch_bounds__(kSumElems * kSumSplit) k_grad_sum(const P *gpart, int nparts, int gsize,
                                                                    double *out) {
    __shared__ double part[kSumSplit][kSumElems];
    grid_dependency_sync();
    const int el = threadIdx.x % kSumElems, q = threadIdx.x / kSumElems;
    const int e = blockIdx.x * kSumElems + el;
    const int p0 = (int)((long long)q * nparts / kSumSplit), p1 = (int)((long long)(q + 1) * nparts / kSumSplit);
    if constexpr (sizeof(P) == 4) {
        CompSum cs;
        if (e < gsize) {
            int p = p0;
            for (; p + 8 <= p1; p += 8) {
                float v[8];
#pragma unroll
                for (int k = 0; k < 8; ++k) v[k] = __ldcg(gpart + (size_t)(p + k) * gsize + e);
#pragma unroll
                for (int k = 0; k < 8; ++k) cs.add(v[k]);
            }
            for (; p < p1; ++p) cs.add(__ldcg(gpart + (size_t)p * gsize + e));
        }
        part[q][el] = (double)cs.s + (double)cs.c;
    } else {
        double t = 0.0;
        if (e < gsize) {
            int p = p0;
            for (; p + 8 <= p1; p += 8) {
                double v[8];
#pragma unroll
                for (int k = 0; k < 8; ++k) v[k] = __ldcg(gpart + (size_t)(p + k) * gsize + e);
#pragma unroll
                for (int k = 0; k < 8; ++k) t += v[k];
            }
            for (; p < p1; ++p) t += __ldcg(gpart + (size_t)p * gsize + e);
        }
        part[q][el] = t;
    }
    __syncthreads();
    if (q == 0 && e < gsize) {
        double t = part[0][el];
#pragma unroll
        for (int k = 1; k < kSumSplit; ++k) t += part[k][el];
        out[e] = t;
    }
}

// Inclusive scan of x[0..n) into y (forward: prefix sums; backward: suffix sums), accumulated in fp64,
// by one warp, in a fixed order: lane c sums a contiguous chunk, the chunk totals
// are scanned across lanes, then every lane writes its chunk.
__device__ void warp_scan(const double *x, double *y, int n, bool backward) {
    const int lane = threadIdx.x & 31;
    const int chunk = (n + 31) / 32;
    const int b = lane * chunk, e = min(n, b + chunk);
    auto at = [&](int i) { return backward ? n - 1 - i : i; };
    double t = 0.0;  // fp64: the sums over intervals cancel
    for (int i = b; i < e; ++i) t += x[at(i)];
    double incl = t;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const double v = __shfl_up_sync(0xffffffffu, incl, o);
        if (lane >= o) incl += v;
    }
    double run = incl - t;  // exclusive prefix of this chunk
    for (int i = b; i < e; ++i) {
        run += x[at(i)];
        y[at(i)] = run;
    }
}

// Block l < L: hidden units of channel l from prefix and suffix sums of the
// channel's interval histogram.  Block L: dW and db.  With the shared-channel
// MLP every channel reads every hidden unit: block l writes its channel's fc1
// contributions to fc1_part ([dw1 | db1][l][k], fp64), summed by k_mlp_fc1_sum.
// With a non-ReLU activation the partials already hold the MLP gradients
// (summed unit by unit): block l copies channel l's, block 0 the shared fc1's.
// Block L also writes the gate's and the coefficients' gradients.
__global__ void __launch_bounds__(128) k_mlp_grads(TableLayout lay, const char *table, const double *gsum,
                                                   luna_phi_grads grads, double *fc1_part) {
    __shared__ double h[2][kMaxUnits + 1];
    __shared__ double pre[2][kMaxUnits + 1], suf[2][kMaxUnits + 1];  // fp64: dw2 = w1 G1 + b1 G0 cancels
    const int Md = lay.M * lay.d, L = lay.L, hid = lay.hid, nint = lay.nint;
    const float scale = 1.0f / sqrtf((float)lay.M);
    const int *rank = reinterpret_cast<const int *>(table + lay.off_rank);
    const int *utype = reinterpret_cast<const int *>(table + lay.off_utype);
    const float *w1 = reinterpret_cast<const float *>(table + lay.off_w1);
    const float *b1 = reinterpret_cast<const float *>(table + lay.off_b1);
    const float *w2 = reinterpret_cast<const float *>(table + lay.off_w2);
    // The first hidden unit of each thread comes from the parameter table, which no kernel of the
    // backward call writes: it is read before the wait for the histogram.
    const bool hist_block = (int)blockIdx.x < L && !lay.act;
    int r_first = 0, t_first = 0;
    float w1_first = 0.0f, b1_first = 0.0f, w2_first = 0.0f;
    if (hist_block && (int)threadIdx.x < hid) {
        const int u = lay.shared ? threadIdx.x : blockIdx.x * hid + threadIdx.x, uw = blockIdx.x * hid + threadIdx.x;
        r_first = rank[u];
        t_first = utype[u];
        w1_first = w1[u];
        b1_first = b1[u];
        w2_first = w2[uw];
    }
    grid_dependency_sync();
    if ((int)blockIdx.x == L) {
        for (int e = threadIdx.x; e < Md; e += blockDim.x) grads.dW[e] = (float)gsum[e];
        for (int e = threadIdx.x; e < lay.M; e += blockDim.x) grads.db[e] = (float)gsum[Md + e];
        const double *gv = gsum + Md + lay.M + mlp_words(lay);  // [dWe | dbe] [dcoef]
        if (lay.env) {
            for (int e = threadIdx.x; e < L * lay.d; e += blockDim.x) grads.dWe[e] = (float)gv[e];
            for (int e = threadIdx.x; e < L; e += blockDim.x) grads.dbe[e] = (float)gv[L * lay.d + e];
            gv += L * lay.d + L;
        }
        if (lay.coef)
            for (int e = threadIdx.x; e < L; e += blockDim.x) grads.dcoef[e] = (float)gv[e];
        return;
    }
    const int l = blockIdx.x;
    const double *hist = gsum + Md + lay.M;
    if (lay.act) {  // [dw2 (L*hid) | dw1 (P) | db1 (P) | db2 (L)]
        const int P = lay.P;
        for (int k = threadIdx.x; k < hid; k += blockDim.x) grads.dw2[l * hid + k] = (float)hist[l * hid + k];
        if (!lay.shared || l == 0) {
            const int u0 = lay.shared ? 0 : l * hid;
            for (int k = threadIdx.x; k < hid; k += blockDim.x) {
                grads.dw1[u0 + k] = (float)hist[L * hid + u0 + k];
                grads.db1[u0 + k] = (float)hist[L * hid + P + u0 + k];
            }
        }
        if (threadIdx.x == 0) grads.db2[l] = (float)hist[L * hid + 2 * P + l];
        return;
    }
    {  // the channel's histogram: every load issued before the first store
        constexpr int kLd = (kMaxUnits + 1 + 127) / 128;
        double v0[kLd], v1[kLd];
#pragma unroll
        for (int k = 0; k < kLd; ++k) {
            const int j = threadIdx.x + 128 * k;
            v0[k] = j < nint ? hist[(j * L + l) * 2] : 0.0;
            v1[k] = j < nint ? hist[(j * L + l) * 2 + 1] : 0.0;
        }
#pragma unroll
        for (int k = 0; k < kLd; ++k) {
            const int j = threadIdx.x + 128 * k;
            if (j < nint) { h[0][j] = v0[k]; h[1][j] = v1[k]; }
        }
    }
    __syncthreads();
    const int warp = threadIdx.x >> 5;  // warps 0, 1: prefix of m0, m1; warps 2, 3: suffix
    warp_scan(h[warp & 1], (warp < 2 ? pre : suf)[warp & 1], nint, warp >= 2);
    __syncthreads();
    for (int k = threadIdx.x; k < hid; k += blockDim.x) {
        const int u = lay.shared ? k : l * hid + k;  // the unit: its kink and fc1
        const int uw = l * hid + k;                  // fc2 weight (l, k)
        const bool first = k == (int)threadIdx.x;
        const int r = first ? r_first : rank[u];
        const bool above = (first ? t_first : utype[u]) > 0;
        const double w1u = first ? w1_first : w1[u], b1u = first ? b1_first : b1[u];
        const double w2u = first ? w2_first : w2[uw];
        double G0, G1;
        if (above) {  // active on intervals j > r
            G0 = r + 1 < nint ? suf[0][r + 1] : 0.0;
            G1 = r + 1 < nint ? suf[1][r + 1] : 0.0;
        } else {      // active on intervals j <= r
            G0 = pre[0][r];
            G1 = pre[1][r];
        }
        grads.dw2[uw] = (float)((w1u * G1 + b1u * G0) * (double)scale);
        const double c1 = w2u * G1 * (double)scale, c0 = w2u * G0 * (double)scale;
        if (lay.shared) {
            fc1_part[(size_t)l * hid + k] = c1;
            fc1_part[(size_t)(L + l) * hid + k] = c0;
        } else {
            grads.dw1[u] = (float)c1;
            grads.db1[u] = (float)c0;
        }
    }
    if (threadIdx.x == 0) grads.db2[l] = (float)(pre[0][nint - 1] * (double)scale);
}

// Shared-channel MLP: dw1[k], db1[k] = sums over the channels (in order) of their contributions.
__global__ void __launch_bounds__(128) k_mlp_fc1_sum(TableLayout lay, const double *fc1_part, luna_phi_grads grads) {
    grid_dependency_sync();
    const int L = lay.L, hid = lay.hid;
    for (int k = threadIdx.x; k < hid; k += blockDim.x) {
        double a = 0.0, b = 0.0;
        for (int l = 0; l < L; ++l) {
            a += fc1_part[(size_t)l * hid + k];
            b += fc1_part[(size_t)(L + l) * hid + k];
        }
        grads.dw1[k] = (float)a;
        grads.db1[k] = (float)b;
    }
}

// ---------------------------------------------------------------------------
// host side

size_t smem_keystats(const AttnArgs &a) {
    HostCarve cv; carve_phi_host(cv, a.lay);
    cv.take(kTileK * a.d); cv.take(kTileK * a.dv); cv.take(kTileK * a.D);
    return cv.bytes();
}
size_t smem_query(const AttnArgs &a) {
    HostCarve cv; carve_phi_host(cv, a.lay);
    cv.take(a.D * a.dv); cv.take(a.D); cv.take(kTileQ * a.d); cv.take(kTileQ * a.D); cv.take(kTileQ);
    return cv.bytes();
}
size_t smem_bwd_query(const AttnArgs &a) {
    HostCarve cv; carve_phi_host(cv, a.lay);
    cv.take(a.D * a.dv); cv.take(a.D); cv.take(kTileB * a.d); cv.take(kTileB * a.dv); cv.take(kTileB * a.D);
    cv.take(kTileB * a.D); cv.take(kTileB * a.dv); cv.take(kTileB); cv.take(kTileB); cv.take(kTileB * a.M);
    cv.take(kTileB * a.M); cv.take(kTileB * a.M);
    return cv.bytes();
}
size_t smem_bwd_key(const AttnArgs &a) {
    HostCarve cv; carve_phi_host(cv, a.lay);
    cv.take(a.D * a.dv); cv.take(a.D); cv.take(kTileB * a.d); cv.take(kTileB * a.dv); cv.take(kTileB * a.D);
    cv.take(kTileB * a.D); cv.take(kTileB * a.M); cv.take(kTileB * a.M); cv.take(kTileB * a.M);
    return cv.bytes();
}

template <typename IO>
cudaError_t stats_impl(const AttnArgs &a, cudaStream_t s) {
    const size_t sm = smem_keystats(a);
    cudaError_t e = set_smem(k_keystats<IO>, sm);
    if (e != cudaSuccess) return e;
    LUNA_LAUNCH("keystats", k_keystats<IO>, dim3(a.nsplit, a.B * a.H), kThreads, sm, s, a);
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
    return launch_chrms_scale_state(a, s);
}

template <typename IO>
cudaError_t fwd_impl(const AttnArgs &a, cudaStream_t s) {
    cudaError_t e = stats_impl<IO>(a, s);
    if (e != cudaSuccess) return e;
    const size_t sm = smem_query(a);
    if ((e = set_smem(k_query<IO>, sm)) != cudaSuccess) return e;
    LUNA_LAUNCH("query", k_query<IO>, dim3((a.n + kTileQ - 1) / kTileQ, a.B * a.H), kThreads, sm, s, a);
    return cudaGetLastError();
}

template <typename IO>
cudaError_t bwd_impl(const AttnArgs &a0, bool have_stats, cudaStream_t s) {
    AttnArgs a = a0;
    a.gpart64 = 1;  // the generic kernels write fp64 parameter-gradient partials
    cudaError_t e;
    if (!have_stats && (e = stats_impl<IO>(a, s)) != cudaSuccess) return e;
    size_t sm = smem_bwd_query(a);
    if ((e = set_smem(k_bwd_query<IO>, sm)) != cudaSuccess) return e;
    LUNA_LAUNCH("bwd_query", k_bwd_query<IO>, dim3(a.nsplit_b, a.B * a.H), kThreads, sm, s, a);
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
    if ((e = launch_chrms_dstate(a, s)) != cudaSuccess) return e;
    sm = smem_bwd_key(a);
    if ((e = set_smem(k_bwd_key<IO>, sm)) != cudaSuccess) return e;
    LUNA_LAUNCH("bwd_key", k_bwd_key<IO>, dim3(a.nsplit_b, a.B * a.H), kThreads, sm, s, a);
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
    int nparts = 0;
    if ((e = launch_chrms_backward(a, 2 * a.B * a.H * a.nsplit_b, &nparts, s)) != cudaSuccess) return e;
    return launch_grad_reduce(a, nparts, s);
}

}  // namespace

size_t simt_max_smem(const AttnArgs &a) {
    size_t m = smem_keystats(a);
    m = m > smem_query(a) ? m : smem_query(a);
    m = m > smem_bwd_query(a) ? m : smem_bwd_query(a);
    m = m > smem_bwd_key(a) ? m : smem_bwd_key(a);
    return m;
}

cudaError_t launch_grad_reduce(const AttnArgs &a, int nparts, cudaStream_t s) {
    const int nb = (a.gsize + kSumElems - 1) / kSumElems;
    const bool dep = !a.ch_sigma;
    if (a.gpart64)
        LUNA_LAUNCH_DEP("grad_sum", dep, k_grad_sum<double>, nb, kSumElems * kSumSplit, 0, s,
                        reinterpret_cast<const double *>(a.gpart), nparts, a.gsize, a.hist);
    else
        LUNA_LAUNCH_DEP("grad_sum", dep, k_grad_sum<float>, nb, kSumElems * kSumSplit, 0, s,
                        static_cast<const float *>(a.gpart), nparts, a.gsize, a.hist);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    if ((e = launch_chrms_hist(a, s)) != cudaSuccess) return e;
    // the partials have been summed: their buffer holds the shared MLP's per-channel fc1 terms
    double *fc1_part = reinterpret_cast<double *>(a.gpart);
    LUNA_LAUNCH_DEP("mlp_grads", dep, k_mlp_grads, a.lay.L + 1, 128, 0, s, a.lay, a.table,
                    static_cast<const double *>(a.hist), a.grads, fc1_part);
    if ((e = cudaGetLastError()) != cudaSuccess || !a.lay.shared || a.lay.act) return e;
    LUNA_LAUNCH_DEP("mlp_fc1_sum", dep, k_mlp_fc1_sum, 1, 128, 0, s, a.lay, static_cast<const double *>(fc1_part),
                    a.grads);
    return cudaGetLastError();
}

cudaError_t launch_featmap(const TableLayout &lay, const char *table, const void *X, luna_dtype xt, int64_t rows,
                           float *Phi, cudaStream_t s) {
    if (lay_variant(lay)) {
        HostCarve cv; carve_phi_host(cv, lay);
        cv.take(kPhiRows * lay.d); cv.take(kPhiRows * lay.D);
        const size_t sm = cv.bytes();
        const int64_t tiles = (rows + kPhiRows - 1) / kPhiRows;
        const int blocks = (int)(tiles < 4096 ? (tiles > 0 ? tiles : 1) : 4096);
        cudaError_t e;
        if (xt == LUNA_F32) {
            if ((e = set_smem(k_featmap_var<float>, sm)) != cudaSuccess) return e;
            k_featmap_var<float><<<blocks, kThreads, sm, s>>>(lay, table, static_cast<const float *>(X), rows, Phi);
        } else {
            if ((e = set_smem(k_featmap_var<__nv_bfloat16>, sm)) != cudaSuccess) return e;
            k_featmap_var<__nv_bfloat16><<<blocks, kThreads, sm, s>>>(lay, table, static_cast<const __nv_bfloat16 *>(X),
                                                                      rows, Phi);
        }
        return cudaGetLastError();
    }
    HostCarve cv; carve_phi_host(cv, lay);
    const size_t sm = cv.bytes();
    int64_t work = rows * lay.M;
    int blocks = (int)((work + kThreads - 1) / kThreads);
    if (blocks > 4096) blocks = 4096;
    if (blocks < 1) blocks = 1;
    cudaError_t e;
    if (xt == LUNA_F32) {
        if ((e = set_smem(k_featmap<float>, sm)) != cudaSuccess) return e;
        k_featmap<float><<<blocks, kThreads, sm, s>>>(lay, table, static_cast<const float *>(X), rows, Phi);
    } else {
        if ((e = set_smem(k_featmap<__nv_bfloat16>, sm)) != cudaSuccess) return e;
        k_featmap<__nv_bfloat16><<<blocks, kThreads, sm, s>>>(lay, table, static_cast<const __nv_bfloat16 *>(X),
                                                              rows, Phi);
    }
    return cudaGetLastError();
}

cudaError_t launch_simt_stats(const AttnArgs &a, luna_dtype io, cudaStream_t s) {
    return io == LUNA_F32 ? stats_impl<float>(a, s) : stats_impl<__nv_bfloat16>(a, s);
}
cudaError_t launch_simt_fwd(const AttnArgs &a, luna_dtype io, cudaStream_t s) {
    return io == LUNA_F32 ? fwd_impl<float>(a, s) : fwd_impl<__nv_bfloat16>(a, s);
}
cudaError_t launch_simt_bwd(const AttnArgs &a, luna_dtype io, bool have_stats, cudaStream_t s) {
    return io == LUNA_F32 ? bwd_impl<float>(a, have_stats, s) : bwd_impl<__nv_bfloat16>(a, have_stats, s);
}

}  // namespace luna
