// Channel RMS normalisation of the feature map (the listing's MLPLearnableFeatureMap
// with ch_rms on), non-causal form.  Each call of the feature map (once over the
// queries, once over the keys) scales channel l of its MLP outputs y_l by
//     s_l = min(target / (rms_l + 1e-6), 1),   rms_l = sqrt(mean y_l^2 + 1e-6),
// the mean over every valid row and projection of that input (a reduction over
// the whole batch).
//
// The attention kernels stay as they are: with phi the unnormalised map, the
// kernel value of Eq. (kernel-attn) is sum_f sigma_l(f) phi_f(q) phi_f(k) with
// sigma_l = s^q_l s^k_l (s >= 0 commutes with the outer ReLU).  So
//   forward:  S, z from the unnormalised keys, rows f scaled by sigma_l(f), then
//             the query pass as before;
//   backward: the query-side kernel (reading the scaled S, z) gives dLoss/dphi(q)
//             of the unnormalised map directly; dS, dz scaled by sigma before the
//             key-side kernel give dLoss/dphi(k) and dV.  Those are the gradients
//             with s held fixed.  The dependence of s_l on every sample adds
//             kappa_l y_l to dLoss/dy_l of every sample of the side, with
//                 kappa_l = ds_l/drms_l * A_l / (N rms_l),
//                 A_l = sum over the side's samples of dLoss/dy_l * y_l / s_l ... (*)
//             and for the non-causal form (*) times s_l equals, on both sides,
//                 T_l = sum_heads sum_{f in channel l} (S'_f . dS_f + z'_f dz_f)
//             (S', z' the scaled statistics, dS, dz before scaling): the sample
//             sums of phi(q) dphi(q) and phi(k) dphi(k) collapse onto the head's
//             statistics.  The kappa term then runs through the ordinary chain
//             rule of the feature map as dLoss/dphi = M kappa_l phi (phi = y/sqrt(M)).
#include <math.h>

#include "luna_prof.cuh"
#include "luna_simt_dev.cuh"

namespace luna {

using namespace simt;

namespace {

constexpr int kRed = 256;          // threads of the one-block reductions (a power of two)
constexpr double kChEps = 1e-6;    // the listing's eps, inside and outside the square root

// Sum of one value per thread in a fixed order (tree over the threads), fp64.
__device__ double block_sum(double v, double *sh) {
    sh[threadIdx.x] = v;
    __syncthreads();
    for (int o = blockDim.x / 2; o > 0; o >>= 1) {
        if ((int)threadIdx.x < o) sh[threadIdx.x] += sh[threadIdx.x + o];
        __syncthreads();
    }
    const double r = sh[0];
    __syncthreads();
    return r;
}

// Sum of phi^2 per channel over the valid rows of one (split, head) block of X (Q or K) and
// every projection: part[(bh * nsplit_b + split) * L + l].
template <typename IO>
__global__ void __launch_bounds__(kThreads) k_chrms_stats(AttnArgs a, const void *Xv, float *part) {
    extern __shared__ __align__(16) float smem[];
    Carve cv{smem};
    const TableLayout &lay = a.lay;
    const int D = a.D, d = a.d, M = a.M, L = a.L;
    SmemPhi s = carve_phi(cv, lay);
    float *sX = cv.take(kTileK * d);
    float *sPhi = cv.take(kTileK * D);
    float *sred = cv.take(kThreads);
    load_phi(s, lay, a.table);
    const int bh = blockIdx.y, split = blockIdx.x;
    const int len = head_length(a.lengths, bh / a.H, a.n);
    const int r0 = split * a.rows_per_split_b;
    const int r1 = min(len, min(a.n, r0 + a.rows_per_split_b));
    const IO *X = static_cast<const IO *>(Xv) + (size_t)bh * a.n * d;
    float acc[kMaxL];
#pragma unroll
    for (int l = 0; l < kMaxL; ++l) acc[l] = 0.0f;
    for (int t0 = r0; t0 < r1; t0 += kTileK) {
        const int nr = min(kTileK, r1 - t0);
        __syncthreads();
        load_rows(sX, X + (size_t)t0 * d, nr * d);
        __syncthreads();
        phi_tile(lay, s, sX, nr, sPhi, nullptr, nullptr);
        __syncthreads();
        for (int e = threadIdx.x; e < nr * M; e += blockDim.x) {  // (row, projection) e: features e*L + l
            const float *ph = sPhi + (size_t)e * L;
#pragma unroll
            for (int l = 0; l < kMaxL; ++l)
                if (l < L) acc[l] = fmaf(ph[l], ph[l], acc[l]);
        }
    }
#pragma unroll
    for (int l = 0; l < kMaxL; ++l) {
        if (l >= L) break;
        __syncthreads();
        sred[threadIdx.x] = acc[l];
        __syncthreads();
        for (int o = blockDim.x / 2; o > 0; o >>= 1) {
            if ((int)threadIdx.x < o) sred[threadIdx.x] += sred[threadIdx.x + o];
            __syncthreads();
        }
        if (threadIdx.x == 0) part[((size_t)bh * a.nsplit_b + split) * L + l] = sred[0];
    }
}

// Statistics of both sides from the block partials (ordered sums, fp64):
// stat[(side*4 + 0..2)*kMaxL + l] = s_l, rms_l, target/(rms_l + eps); stat[3*kMaxL] = N
// (samples per side: valid rows x M); sigma[l] = s^q_l s^k_l.
__global__ void __launch_bounds__(kRed) k_chrms_scales(AttnArgs a, const float *part, int nparts, float target,
                                                       double *stat, float *sigma) {
    __shared__ double sh[kRed];
    const int BH = a.B * a.H, L = a.L;
    double rows = 0.0;
    for (int bh = threadIdx.x; bh < BH; bh += blockDim.x) rows += head_length(a.lengths, bh / a.H, a.n);
    const double N = block_sum(rows, sh) * a.M;
    for (int side = 0; side < 2; ++side)
        for (int l = 0; l < L; ++l) {
            double v = 0.0;
            for (int p = threadIdx.x; p < nparts; p += blockDim.x) v += part[((size_t)side * nparts + p) * L + l];
            v = block_sum(v, sh);
            if (threadIdx.x == 0) {
                const double mean = N > 0.0 ? v * a.M / N : 0.0;  // y = sqrt(M) phi
                const double rms = sqrt(mean + kChEps);
                const double r = (double)target / (rms + kChEps);
                stat[(side * 4 + 0) * kMaxL + l] = r < 1.0 ? r : 1.0;
                stat[(side * 4 + 1) * kMaxL + l] = rms;
                stat[(side * 4 + 2) * kMaxL + l] = r;
            }
        }
    if (threadIdx.x == 0) stat[3 * kMaxL] = N;
    __syncthreads();
    if ((int)threadIdx.x < L) sigma[threadIdx.x] = (float)(stat[threadIdx.x] * stat[4 * kMaxL + threadIdx.x]);
}

// rows f of S [BH][D][dv] and z [BH][D] times sigma_{f mod L}
__global__ void k_chrms_scale_rows(float *S, float *z, const float *sigma, int64_t BH, int D, int L, int dv) {
    const int64_t nS = BH * D * dv, nz = BH * D;
    const int64_t step = (int64_t)gridDim.x * blockDim.x;
    for (int64_t e = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; e < nS; e += step)
        S[e] *= sigma[(int)((e / dv) % D) % L];
    for (int64_t e = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; e < nz; e += step) z[e] *= sigma[(int)(e % D) % L];
}

// Per head: T[bh][l] = sum_{f in channel l} (S'_f . dS_f + z'_f dz_f), then dS, dz rows times sigma.
__global__ void __launch_bounds__(128) k_chrms_dstate(AttnArgs a, const float *sigma, double *T) {
    __shared__ float dots[kMaxFeat];
    const int bh = blockIdx.x, D = a.D, dv = a.dv, L = a.L;
    const float *S = a.S_fin + (size_t)bh * D * dv;
    const float *z = a.z_fin + (size_t)bh * D;
    float *G = a.dS_fin + (size_t)bh * D * dv;
    float *g = a.dz_fin + (size_t)bh * D;
    for (int f = threadIdx.x; f < D; f += blockDim.x) {
        float t = z[f] * g[f];
        for (int c = 0; c < dv; ++c) t = fmaf(S[(size_t)f * dv + c], G[(size_t)f * dv + c], t);
        dots[f] = t;
        const float sg = sigma[f % L];
        for (int c = 0; c < dv; ++c) G[(size_t)f * dv + c] *= sg;
        g[f] *= sg;
    }
    __syncthreads();
    if ((int)threadIdx.x < L) {
        double t = 0.0;
        for (int f = threadIdx.x; f < D; f += L) t += dots[f];
        T[(size_t)bh * L + threadIdx.x] = t;
    }
}

// kappa[side*kMaxL + l] = d s_l / d rms_l * (T_l / s_l) / (N rms_l), zero where the scale is clamped
// at 1 (target/(rms + eps) > 1) or the side has no samples.
__global__ void __launch_bounds__(kRed) k_chrms_kappa(AttnArgs a, const double *T, float target, const double *stat,
                                                      float *kappa) {
    __shared__ double sh[kRed];
    const int BH = a.B * a.H, L = a.L;
    const double N = stat[3 * kMaxL];
    for (int l = 0; l < L; ++l) {
        double v = 0.0;
        for (int bh = threadIdx.x; bh < BH; bh += blockDim.x) v += T[(size_t)bh * L + l];
        v = block_sum(v, sh);
        if (threadIdx.x == 0)
            for (int side = 0; side < 2; ++side) {
                const double s = stat[(side * 4 + 0) * kMaxL + l], rms = stat[(side * 4 + 1) * kMaxL + l];
                const double r = stat[(side * 4 + 2) * kMaxL + l];
                const double ds = -(double)target / ((rms + kChEps) * (rms + kChEps));  // d s / d rms, unclamped
                kappa[side * kMaxL + l] = (N > 0.0 && r <= 1.0) ? (float)(ds * (v / s) / (N * rms)) : 0.0f;
            }
    }
}

template <typename IO>
__device__ void add_dx(const TableLayout &lay, const SmemPhi &s, const float *sdU, int nr, IO *dX) {
    const int M = lay.M, d = lay.d;
    for (int e = threadIdx.x; e < nr * d; e += blockDim.x) {
        const int r = e / d, c = e - r * d;
        float acc = io_load(dX + e);
        for (int i = 0; i < M; ++i) acc = fmaf(sdU[r * M + i], s.W[i * d + c], acc);
        io_store(dX + e, acc);
    }
}

// The kappa term of one side: dLoss/dphi = M kappa_l phi on every valid sample, through the
// chain rule of the (unnormalised) feature map; adds to dQ or dK and writes one parameter-gradient
// partial per (split, head) block at gpart[(side * BH * nsplit_b + bh * nsplit_b + split) * gsize].
template <typename IO>
__global__ void __launch_bounds__(kThreads) k_chrms_phi_bwd(AttnArgs a, int side, const float *kappa, float *gpart) {
    extern __shared__ __align__(16) float smem[];
    Carve cv{smem};
    const TableLayout &lay = a.lay;
    const int D = a.D, d = a.d, M = a.M, L = a.L;
    SmemPhi s = carve_phi(cv, lay);
    float *sX = cv.take(kTileB * d);
    float *sPhi = cv.take(kTileB * D);
    float *sdPhi = cv.take(kTileB * D);
    float *sU = cv.take(kTileB * M);
    int *sJ = reinterpret_cast<int *>(cv.take(kTileB * M));
    float *sdU = cv.take(kTileB * M);
    float *shist = cv.take(lay.nint * L * 2);
    float *sk = cv.take(kMaxL);
    load_phi(s, lay, a.table);
    for (int e = threadIdx.x; e < lay.nint * L * 2; e += blockDim.x) shist[e] = 0.0f;
    if ((int)threadIdx.x < L) sk[threadIdx.x] = kappa[side * kMaxL + threadIdx.x] * (float)M;
    const int bh = blockIdx.y, split = blockIdx.x;
    const int len = head_length(a.lengths, bh / a.H, a.n);
    const int r0 = split * a.rows_per_split_b;
    const int r1 = min(len, min(a.n, r0 + a.rows_per_split_b));
    const IO *X = static_cast<const IO *>(side ? a.K : a.Q) + (size_t)bh * a.n * d;
    IO *dX = static_cast<IO *>(side ? a.dK : a.dQ) + (size_t)bh * a.n * d;
    GradAcc g = {};
    for (int t0 = r0; t0 < r1; t0 += kTileB) {
        const int nr = min(kTileB, r1 - t0);
        __syncthreads();
        load_rows(sX, X + (size_t)t0 * d, nr * d);
        __syncthreads();
        phi_tile(lay, s, sX, nr, sPhi, sU, sJ);
        __syncthreads();
        for (int e = threadIdx.x; e < nr * D; e += blockDim.x) sdPhi[e] = sk[e % L] * sPhi[e];  // D = M*L
        __syncthreads();
        phi_backward_tile(lay, s, sX, nr, sPhi, sdPhi, sU, sJ, sdU, shist, g);
        add_dx(lay, s, sdU, nr, dX + (size_t)t0 * d);
    }
    __syncthreads();
    const size_t slot = (size_t)side * a.B * a.H * a.nsplit_b + (size_t)bh * a.nsplit_b + split;
    store_grad_partial(lay, g, shist, gpart + slot * a.gsize);
}

size_t smem_stats(const AttnArgs &a) {
    HostCarve cv; carve_phi_host(cv, a.lay);
    cv.take(kTileK * a.d); cv.take(kTileK * a.D); cv.take(kThreads);
    return cv.bytes();
}
size_t smem_phi_bwd(const AttnArgs &a) {
    HostCarve cv; carve_phi_host(cv, a.lay);
    cv.take(kTileB * a.d); cv.take(kTileB * a.D); cv.take(kTileB * a.D);
    cv.take(kTileB * a.M); cv.take(kTileB * a.M); cv.take(kTileB * a.M);
    cv.take(a.lay.nint * a.lay.L * 2); cv.take(kMaxL);
    return cv.bytes();
}

template <typename IO>
cudaError_t stats_impl(const AttnArgs &a, cudaStream_t s) {
    const int nparts = a.B * a.H * a.nsplit_b;
    const size_t sm = smem_stats(a);
    cudaError_t e = set_smem(k_chrms_stats<IO>, sm);
    if (e != cudaSuccess) return e;
    for (int side = 0; side < 2; ++side) {
        LUNA_LAUNCH("chrms_stats", k_chrms_stats<IO>, dim3(a.nsplit_b, a.B * a.H), kThreads, sm, s, a,
                    side ? a.K : a.Q, a.ch_part + (size_t)side * nparts * a.L);
        if ((e = cudaGetLastError()) != cudaSuccess) return e;
    }
    LUNA_LAUNCH("chrms_scales", k_chrms_scales, 1, kRed, 0, s, a, a.ch_part, nparts, a.ch_target, a.ch_stat,
                a.ch_sigma);
    return cudaGetLastError();
}

template <typename IO>
cudaError_t phi_bwd_impl(const AttnArgs &a, float *gpart, cudaStream_t s) {
    const size_t sm = smem_phi_bwd(a);
    cudaError_t e = set_smem(k_chrms_phi_bwd<IO>, sm);
    if (e != cudaSuccess) return e;
    for (int side = 0; side < 2; ++side) {
        LUNA_LAUNCH("chrms_phi_bwd", k_chrms_phi_bwd<IO>, dim3(a.nsplit_b, a.B * a.H), kThreads, sm, s, a, side,
                    a.ch_kappa, gpart);
        if ((e = cudaGetLastError()) != cudaSuccess) return e;
    }
    return cudaSuccess;
}

int blocks_for(int64_t n) {
    const int64_t b = (n + 255) / 256;
    return (int)(b < 1 ? 1 : (b > 4096 ? 4096 : b));
}

}  // namespace

size_t chrms_max_smem(const AttnArgs &a) {
    const size_t x = smem_stats(a), y = smem_phi_bwd(a);
    return x > y ? x : y;
}

cudaError_t launch_chrms_stats(const AttnArgs &a, luna_dtype io, cudaStream_t s) {
    return io == LUNA_F32 ? stats_impl<float>(a, s) : stats_impl<__nv_bfloat16>(a, s);
}

cudaError_t launch_chrms_scale_state(const AttnArgs &a, cudaStream_t s) {
    if (!a.ch_sigma) return cudaSuccess;
    const int64_t BH = (int64_t)a.B * a.H;
    LUNA_LAUNCH("chrms_scale", k_chrms_scale_rows, blocks_for(BH * a.D * a.dv), 256, 0, s, a.S_fin, a.z_fin,
                a.ch_sigma, BH, a.D, a.L, a.dv);
    return cudaGetLastError();
}

cudaError_t launch_chrms_dstate(const AttnArgs &a, cudaStream_t s) {
    if (!a.ch_sigma) return cudaSuccess;
    LUNA_LAUNCH("chrms_dstate", k_chrms_dstate, a.B * a.H, 128, 0, s, a, a.ch_sigma, a.ch_T);
    return cudaGetLastError();
}

cudaError_t launch_chrms_backward(const AttnArgs &a, int main_parts, int *nparts, cudaStream_t s) {
    *nparts = main_parts;
    if (!a.ch_sigma) return cudaSuccess;
    LUNA_LAUNCH("chrms_kappa", k_chrms_kappa, 1, kRed, 0, s, a, a.ch_T, a.ch_target, a.ch_stat, a.ch_kappa);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    float *gpart = a.gpart + (size_t)main_parts * a.gsize;
    e = a.ch_io == LUNA_F32 ? phi_bwd_impl<float>(a, gpart, s) : phi_bwd_impl<__nv_bfloat16>(a, gpart, s);
    if (e != cudaSuccess) return e;
    *nparts = main_parts + 2 * a.B * a.H * a.nsplit_b;
    return cudaSuccess;
}

}  // namespace luna
