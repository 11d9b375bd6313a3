// Channel RMS normalisation of the feature map (the listing's MLPLearnableFeatureMap
// with ch_rms on), non-causal form.  Each call of the feature map (once over the
// queries, once over the keys) scales channel l of its MLP outputs y_l by
//     s_l = min(target / (rms_l + 1e-6), 1),   rms_l = sqrt(mean y_l^2 + 1e-6),
// the mean over every valid row and projection of that input (a reduction over
// the whole batch).
//
// The attention kernels stay as they are.  With phi the unnormalised map, the
// kernel value of Eq. (kernel-attn) is sum_f sigma_l(f) phi_f(q) phi_f(k) with
// sigma_l = s^q_l s^k_l (s >= 0 commutes with the outer ReLU).  So
//   forward:  S, z from the unnormalised keys, rows f scaled by sigma_l(f), then
//             the query pass as before;
//   backward: the query-side kernel, reading the scaled S, z, gives dLoss/dphi(q)
//             of the unnormalised map directly; dS, dz scaled by sigma before the
//             key-side kernel give dLoss/dphi(k) and dV.  These are the gradients
//             with s held fixed.
// The dependence of s_l on every sample of a side adds kappa_l y_l to dLoss/dy_l
// of each of that side's samples, where
//     kappa_l = ds_l/drms_l * A_l / (N rms_l),   ds_l/drms_l = -target / (rms_l + 1e-6)^2
// (zero where s_l is clamped at 1), N the side's sample count and A_l the sum over
// the side's samples of y_l times dLoss/d(s_l y_l).  For the non-causal form
//     s_l A_l = T_l = sum over heads and the channel's feature rows f of (S'_f . dS_f + z'_f dz_f)
// on both sides (S', z' the scaled statistics, dS, dz before scaling): the sample
// sums collapse onto each head's statistics.  The kappa term then runs through the
// ordinary chain rule of the feature map as dLoss/dphi = M kappa_l phi (phi = y/sqrt(M)).
//
// Streaming (causal) form: the prefix states do not collapse the sample sums, so
// both sides run on a copy of the table whose channel-l coefficients are scaled
// by sqrt(sigma_l): phi^ = sqrt(sigma) phi on queries and keys gives the same
// kernel value, and the streaming kernels run unchanged.  T_l is the sum over the
// query samples of phi^ . dLoss/dphi^ on channel l (equal to the sum over the
// normalised features, and the same for the key side, since the loss depends on
// s^q_l and s^k_l only through their product): the tensor-core query sweep sums
// it where it forms dphi^(q), so kappa is known before either chain rule, which
// adds M (kappa_l / sigma_l) phi^ to dLoss/dphi^ (its dU is then that of the
// unscaled map's scale term); the generic path sums T in its query-side kernel
// and runs the kappa pass on the scaled table with kappa_l / sigma_l.  Before
// the channel-MLP gradients the reduced interval histogram of channel l, a sum
// of dLoss/dphi^, is multiplied by sqrt(sigma_l) to give sums of dLoss/dphi.
#include <math.h>

#include "luna_prof.cuh"
#include "luna_simt_dev.cuh"

namespace luna {

using namespace simt;

namespace {

constexpr int kRed = 256;          // threads of the one-block reductions (a power of two)
constexpr int kKWarps = 4;         // warps per block of the kappa-term pass
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

// Sum of phi^2 per channel over the valid rows and every projection of one side (blockIdx.y: 0 = Q,
// 1 = K): one thread per row in a grid-stride loop, all M projections of the row in registers, no block
// barriers in the loop; block partials at part[(side * gridDim.x + blockIdx.x) * L + l].  W sits
// transposed in shared memory, padded to kStatMP columns (WT[c][i]): every lane of a warp reads the same
// four-word group at once (a broadcast), so the projections cost one shared load per four FMAs.  Each u_i
// is the fp32 chain b_i + sum_c W_ic x_c in order of c; the interval comes from the bucketed search block.
constexpr int kStatMP = 32;  // projections held per row (M <= 32)
template <typename IO, bool VEC>
__global__ void __launch_bounds__(kThreads) k_chrms_stats(AttnArgs a, float *part) {
    extern __shared__ __align__(16) float smem[];
    const TableLayout &lay = a.lay;
    const int d = a.d, M = a.M, L = a.L;
    float *sS = smem;                          // the interval search block
    float *sAB = sS + kEytzinger;
    float *sWT = sAB + r4(lay.nint * ab_stride(lay));  // [d][kStatMP]
    float *sb = sWT + d * kStatMP;             // [kStatMP]
    float *sred = sb + kStatMP;
    {
        const float *S = reinterpret_cast<const float *>(a.table + lay.off_Te);
        const float *W = reinterpret_cast<const float *>(a.table + lay.off_W);
        const float *b = reinterpret_cast<const float *>(a.table + lay.off_b);
        for (int e = threadIdx.x; e < kEytzinger; e += blockDim.x) sS[e] = S[e];
        copy_ab(sAB, lay, a.table);
        for (int e = threadIdx.x; e < d * kStatMP; e += blockDim.x) {
            const int c = e / kStatMP, i = e - c * kStatMP;
            sWT[e] = i < M ? W[i * d + c] : 0.0f;
        }
        for (int e = threadIdx.x; e < kStatMP; e += blockDim.x) sb[e] = e < M ? b[e] : 0.0f;
    }
    __syncthreads();
    const unsigned short *sB = reinterpret_cast<const unsigned short *>(sS + kSearchT);
    const int side = blockIdx.y;
    const IO *X = static_cast<const IO *>(side ? a.K : a.Q);
    const int64_t rows = (int64_t)a.B * a.H * a.n;
    float acc[kMaxL];
#pragma unroll
    for (int l = 0; l < kMaxL; ++l) acc[l] = 0.0f;
    // the projections of one input column: u_i += W_ic x_c for the groups of four with a live projection
    auto column = [&](float (&u)[kStatMP], int c, float xc) {
        const float4 *w = reinterpret_cast<const float4 *>(sWT + c * kStatMP);
#pragma unroll
        for (int q = 0; q < kStatMP / 4; ++q)
            if (4 * q < M) {
                const float4 ww = w[q];
                u[4 * q] = fmaf(ww.x, xc, u[4 * q]);
                u[4 * q + 1] = fmaf(ww.y, xc, u[4 * q + 1]);
                u[4 * q + 2] = fmaf(ww.z, xc, u[4 * q + 2]);
                u[4 * q + 3] = fmaf(ww.w, xc, u[4 * q + 3]);
            }
    };
    for (int64_t row = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; row < rows;
         row += (int64_t)gridDim.x * blockDim.x) {
        const int64_t bh = row / a.n;
        if ((int)(row - bh * a.n) >= head_length(a.lengths, (int)(bh / a.H), a.n)) continue;
        const IO *x = X + row * d;
        float u[kStatMP];
#pragma unroll
        for (int i = 0; i < kStatMP; ++i) u[i] = sb[i];
        if (VEC) {  // 16-byte loads: 8 bf16 or 4 fp32 values
            constexpr int V = 16 / sizeof(IO);
            for (int c0 = 0; c0 < d; c0 += V) {
                const uint4 raw = __ldg(reinterpret_cast<const uint4 *>(x + c0));
                const IO *v = reinterpret_cast<const IO *>(&raw);
#pragma unroll
                for (int k = 0; k < V; ++k) column(u, c0 + k, io_load(v + k));
            }
        } else {
            for (int c = 0; c < d; ++c) column(u, c, io_load(x + c));
        }
#pragma unroll
        for (int i = 0; i < kStatMP; ++i) {
            if (i >= M) break;
            const float *ab = sAB + interval_bucketed(sS, sB, u[i]) * ab_stride(lay);
#pragma unroll
            for (int l = 0; l < kMaxL; ++l)
                if (l < L) {
                    const float2 p = ab_pair(ab, l);
                    const float y = fmaxf(fmaf(p.x, u[i], p.y), 0.0f);
                    acc[l] = fmaf(y, y, acc[l]);
                }
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
        if (threadIdx.x == 0) part[((size_t)side * gridDim.x + blockIdx.x) * L + l] = sred[0];
    }
}

// Sum over p < n of x[p * stride] by one warp, lanes over p, then a fixed shuffle tree (fp64).
__device__ double warp_sum_strided(const float *x, int n, int stride) {
    const int lane = threadIdx.x & 31;
    double v = 0.0;
    for (int p = lane; p < n; p += 32) v += x[(size_t)p * stride];
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    return v;
}

// Statistics of both sides from the block partials (fixed-order sums, fp64), one warp per
// (side, channel): stat[(side*4 + 0..2)*kMaxL + l] = s_l, rms_l, target/(rms_l + eps);
// stat[3*kMaxL] = N (samples per side: valid rows x M); sigma[l] = s^q_l s^k_l.
__global__ void __launch_bounds__(kRed) k_chrms_scales(AttnArgs a, const float *part, int nparts, float target,
                                                       double *stat, float *sigma) {
    __shared__ double sh[kRed];
    __shared__ double ssc[2 * kMaxL];
    const int BH = a.B * a.H, L = a.L, warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    double rows = 0.0;
    for (int bh = threadIdx.x; bh < BH; bh += blockDim.x) rows += head_length(a.lengths, bh / a.H, a.n);
    const double N = block_sum(rows, sh) * a.M;
    for (int q = warp; q < 2 * L; q += blockDim.x >> 5) {
        const int side = q / L, l = q - side * L;
        const double v = warp_sum_strided(part + (size_t)side * nparts * L + l, nparts, L);
        if (lane == 0) {
            const double mean = N > 0.0 ? v * a.M / N : 0.0;  // y = sqrt(M) phi
            const double rms = sqrt(mean + kChEps);
            const double r = (double)target / (rms + kChEps);
            const double sl = r < 1.0 ? r : 1.0;
            stat[(side * 4 + 0) * kMaxL + l] = sl;
            stat[(side * 4 + 1) * kMaxL + l] = rms;
            stat[(side * 4 + 2) * kMaxL + l] = r;
            ssc[side * kMaxL + l] = sl;
        }
    }
    if (threadIdx.x == 0) stat[3 * kMaxL] = N;
    __syncthreads();
    if ((int)threadIdx.x < L) sigma[threadIdx.x] = (float)(ssc[threadIdx.x] * ssc[kMaxL + threadIdx.x]);
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
// at 1 (target/(rms + eps) > 1) or the side has no samples; T_l the sum of rows T[0 .. BH)[l] in order.
// With `sigma` (the streaming form's scaled table), kappa_l / sigma_l.
__global__ void __launch_bounds__(kRed) k_chrms_kappa(AttnArgs a, const double *T, int BH, float target,
                                                      const double *stat, const float *sigma, float *kappa) {
    const int L = a.L, warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const double N = stat[3 * kMaxL];
    for (int l = warp; l < L; l += blockDim.x >> 5) {
        double v = 0.0;
        for (int bh = lane; bh < BH; bh += 32) v += T[(size_t)bh * L + l];
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
        if (lane == 0)
            for (int side = 0; side < 2; ++side) {
                const double s = stat[(side * 4 + 0) * kMaxL + l], rms = stat[(side * 4 + 1) * kMaxL + l];
                const double r = stat[(side * 4 + 2) * kMaxL + l];
                const double ds = -(double)target / ((rms + kChEps) * (rms + kChEps));  // d s / d rms, unclamped
                const double k = (N > 0.0 && r <= 1.0) ? ds * (v / s) / (N * rms) : 0.0;
                kappa[side * kMaxL + l] = (float)(sigma ? k / (double)sigma[l] : k);
            }
    }
}

// The kappa term of both sides (blockIdx.y: 0 = Q, 1 = K): dLoss/dphi = M kappa_l phi on every valid
// sample, through the chain rule of the unnormalised feature map.  Each warp takes 32 consecutive rows
// (lane = row) in a grid-stride loop: it stages them in shared memory (row stride d + 1, so the lanes'
// rows fall in distinct banks), computes every projection's u, interval, channels and dU, then, with
// the lanes over input columns, adds dU W to the rows of dQ / dK and dU^T X, column sums of dU to the
// block's dW, db.  One parameter-gradient partial per block at gpart[(side * gridDim.x + blockIdx.x) *
// gsize], of the partials' type P (fp32 beside the tensor-core kernels' partials, fp64 beside the
// generic kernels'); its interval histogram is accumulated in place by reductions in L2 (atomic adds
// without a return value), which do not serialise like fp32 atomics in shared memory.
template <typename IO, typename GP>
__global__ void __launch_bounds__(kKWarps * 32) k_chrms_kterm(AttnArgs a, const float *kappa, GP *gpart) {
    extern __shared__ __align__(16) float smem[];
    const TableLayout &lay = a.lay;
    const int d = a.d, M = a.M, L = a.L, P = lay.Ppad, NH = lay.nint * L * 2;
    const int dp = d + 1, mp = M + 1;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int side = blockIdx.y;
    float *sT = smem;
    float *sAB = sT + r4(P);
    float *sW = sAB + r4(lay.nint * ab_stride(lay));
    float *sb = sW + r4(M * d);
    GP *sdW = reinterpret_cast<GP *>(sb + r4(M));  // block sums of dW, db in the partials' type
    GP *sdb = sdW + r4(M * d);
    float *sk = reinterpret_cast<float *>(sdb + r4(M));
    float *sx = sk + r4(kMaxL) + warp * (r4(32 * dp) + r4(32 * mp));
    float *sdu = sx + r4(32 * dp);
    if (!carve_fits(Carve{sk + r4(kMaxL) + kKWarps * (r4(32 * dp) + r4(32 * mp))}, smem)) return;
    const int Md = M * d;
    GP *gp = gpart + ((size_t)side * gridDim.x + blockIdx.x) * a.gsize;
    GP *ghist = gp + Md + M;
    {
        const float *T = reinterpret_cast<const float *>(a.table + lay.off_T);
        const float *W = reinterpret_cast<const float *>(a.table + lay.off_W);
        const float *b = reinterpret_cast<const float *>(a.table + lay.off_b);
        for (int e = threadIdx.x; e < P; e += blockDim.x) sT[e] = T[e];
        copy_ab(sAB, lay, a.table);
        for (int e = threadIdx.x; e < NH; e += blockDim.x) ghist[e] = (GP)0;
        for (int e = threadIdx.x; e < M * d; e += blockDim.x) { sW[e] = W[e]; sdW[e] = (GP)0; }
        for (int e = threadIdx.x; e < M; e += blockDim.x) { sb[e] = b[e]; sdb[e] = (GP)0; }
        if ((int)threadIdx.x < L) sk[threadIdx.x] = kappa[side * kMaxL + threadIdx.x] * (float)M;
    }
    __syncthreads();
    const IO *X = static_cast<const IO *>(side ? a.K : a.Q);
    IO *dX = static_cast<IO *>(side ? a.dK : a.dQ);
    const int64_t rows = (int64_t)a.B * a.H * a.n;
    const int64_t ngroups = (rows + 31) / 32;
    for (int64_t grp = (int64_t)blockIdx.x * kKWarps + warp; grp < ngroups; grp += (int64_t)gridDim.x * kKWarps) {
        const int64_t row0 = grp * 32, myrow = row0 + lane;
        bool valid = false;
        if (myrow < rows) {
            const int64_t bh = myrow / a.n;
            valid = (int)(myrow - bh * a.n) < head_length(a.lengths, (int)(bh / a.H), a.n);
        }
        const unsigned vmask = __ballot_sync(0xffffffffu, valid);
        if (vmask == 0u) continue;
        for (int r = 0; r < 32; ++r) {
            const bool vr = (vmask >> r) & 1u;
            for (int c = lane; c < d; c += 32) sx[r * dp + c] = vr ? io_load(X + (row0 + r) * d + c) : 0.0f;
        }
        __syncwarp();
        for (int i = 0; i < M; ++i) {
            float du = 0.0f;
            if (valid) {
                const float *w = sW + i * d, *x = sx + lane * dp;
                float u = sb[i];
                for (int c = 0; c < d; ++c) u = fmaf(w[c], x[c], u);
                const int j = interval_of(sT, P, u);
                const float *ab = sAB + j * ab_stride(lay);
                GP *h = ghist + j * L * 2;
                for (int l = 0; l < L; ++l) {
                    const float2 p = ab_pair(ab, l);
                    const float ph = fmaxf(fmaf(p.x, u, p.y), 0.0f);
                    if (ph > 0.0f) {  // outer ReLU on
                        const float g = sk[l] * ph;
                        du = fmaf(g, p.x, du);
                        if (g != 0.0f) {
                            atomicAdd(h + 2 * l, (GP)g);
                            atomicAdd(h + 2 * l + 1, (GP)g * (GP)u);
                        }
                    }
                }
            }
            sdu[lane * mp + i] = du;
        }
        __syncwarp();
        for (int c = lane; c < d; c += 32) {
            float cur[32];  // the 32 rows' current values, all loaded before any store
#pragma unroll
            for (int r = 0; r < 32; ++r) cur[r] = ((vmask >> r) & 1u) ? io_load(dX + (row0 + r) * d + c) : 0.0f;
#pragma unroll
            for (int r = 0; r < 32; ++r) {
                if (!((vmask >> r) & 1u)) continue;
                float acc = 0.0f;
                for (int i = 0; i < M; ++i) acc = fmaf(sdu[r * mp + i], sW[i * d + c], acc);
                io_store(dX + (row0 + r) * d + c, cur[r] + acc);
            }
            for (int i = 0; i < M; ++i) {
                GP acc = (GP)0;
                for (int r = 0; r < 32; ++r) acc = fma((GP)sdu[r * mp + i], (GP)sx[r * dp + c], acc);
                atomicAdd(sdW + i * d + c, acc);
            }
        }
        if (lane < M) {
            GP acc = (GP)0;
            for (int r = 0; r < 32; ++r) acc += (GP)sdu[r * mp + lane];
            atomicAdd(sdb + lane, acc);
        }
        __syncwarp();
    }
    __syncthreads();
    for (int e = threadIdx.x; e < Md; e += blockDim.x) gp[e] = (GP)sdW[e];
    for (int e = threadIdx.x; e < M; e += blockDim.x) gp[Md + e] = (GP)sdb[e];
}

// Copy of the table with every channel's (alpha, beta) scaled by sqrt(sigma_l) (streaming form).
__global__ void k_chrms_scale_table(const float *src, float *dst, TableLayout lay, const float *sigma) {
    const int64_t n = lay.bytes / 4, ab0 = lay.off_AB / 4, ab1 = ab0 + (int64_t)lay.nint * lay.L * 2;
    for (int64_t e = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; e < n; e += (int64_t)gridDim.x * blockDim.x) {
        float v = src[e];
        if (e >= ab0 && e < ab1) v *= sqrtf(sigma[(int)(((e - ab0) >> 1) % lay.L)]);
        dst[e] = v;
    }
}

// Reduced interval histogram [nint][L][2] (after dW, db) of channel l times sqrt(sigma_l).
__global__ void k_chrms_scale_hist(double *gsum, TableLayout lay, const float *sigma) {
    double *h = gsum + (size_t)lay.M * lay.d + lay.M;
    for (int e = blockIdx.x * blockDim.x + threadIdx.x; e < lay.nint * lay.L * 2; e += gridDim.x * blockDim.x)
        h[e] *= sqrt((double)sigma[(e >> 1) % lay.L]);
}

size_t smem_stats(const AttnArgs &a) {
    return (size_t)(kEytzinger + r4(a.lay.nint * ab_stride(a.lay)) + a.d * kStatMP + kStatMP + kThreads) * 4;
}
// shared memory of the scale-term pass with block sums of GP (gp_words: 4-byte words per GP)
size_t smem_kterm(const AttnArgs &a, int gp_words = 2) {
    return (size_t)(r4(a.lay.Ppad) + r4(a.lay.nint * ab_stride(a.lay)) + (1 + gp_words) * (r4(a.M * a.d) + r4(a.M)) + r4(kMaxL) +
                    kKWarps * (r4(32 * (a.d + 1)) + r4(32 * (a.M + 1)))) * 4;
}

template <typename IO, bool VEC>
cudaError_t stats_impl(const AttnArgs &a, cudaStream_t s) {
    const size_t sm = smem_stats(a);
    cudaError_t e = set_smem(k_chrms_stats<IO, VEC>, sm);
    if (e != cudaSuccess) return e;
    LUNA_LAUNCH("chrms_stats", (k_chrms_stats<IO, VEC>), dim3(kChStatBlocks, 2), kThreads, sm, s, a, a.ch_part);
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
    LUNA_LAUNCH("chrms_scales", k_chrms_scales, 1, kRed, 0, s, a, a.ch_part, kChStatBlocks, a.ch_target, a.ch_stat,
                a.ch_sigma);
    return cudaGetLastError();
}

template <typename IO, typename GP>
cudaError_t kterm_impl(const AttnArgs &a, GP *gpart, cudaStream_t s) {
    const size_t sm = smem_kterm(a, (int)(sizeof(GP) / 4));
    cudaError_t e = set_smem(k_chrms_kterm<IO, GP>, sm);
    if (e != cudaSuccess) return e;
    LUNA_LAUNCH("chrms_kterm", (k_chrms_kterm<IO, GP>), dim3(kChKBlocks, 2), kKWarps * 32, sm, s, a, a.ch_kappa,
                gpart);
    return cudaGetLastError();
}

int blocks_for(int64_t n) {
    const int64_t b = (n + 255) / 256;
    return (int)(b < 1 ? 1 : (b > 4096 ? 4096 : b));
}

}  // namespace

size_t chrms_max_smem(const AttnArgs &a) {
    const size_t x = smem_stats(a), y = smem_kterm(a);
    return x > y ? x : y;
}

bool tc_chstats_supported(const AttnArgs &a, luna_dtype io);
cudaError_t launch_tc_chstats(const AttnArgs &a, float *part, int max_parts, int *nparts, cudaStream_t s);

cudaError_t launch_chrms_stats(const AttnArgs &a, luna_dtype io, cudaStream_t s) {
    if (tc_chstats_supported(a, io)) {  // the projections on tensor cores (luna_tc_chstats.cu)
        int nparts = 0;
        cudaError_t e = launch_tc_chstats(a, a.ch_part, kChStatBlocks, &nparts, s);
        if (e != cudaSuccess) return e;
        LUNA_LAUNCH("chrms_scales", k_chrms_scales, 1, kRed, 0, s, a, a.ch_part, nparts, a.ch_target, a.ch_stat,
                    a.ch_sigma);
        return cudaGetLastError();
    }
    // 16-byte row loads when every row starts on a 16-byte boundary
    const size_t rb = (size_t)a.d * (io == LUNA_F32 ? 4 : 2);
    const bool vec = rb % 16 == 0 && (reinterpret_cast<uintptr_t>(a.Q) & 15) == 0 &&
                     (reinterpret_cast<uintptr_t>(a.K) & 15) == 0;
    if (io == LUNA_F32) return vec ? stats_impl<float, true>(a, s) : stats_impl<float, false>(a, s);
    return vec ? stats_impl<__nv_bfloat16, true>(a, s) : stats_impl<__nv_bfloat16, false>(a, s);
}

cudaError_t launch_chrms_scale_state(const AttnArgs &a, cudaStream_t s) {
    // non-causal only: the streaming form has no S_fin, z_fin (its sigma sits in the scaled table)
    if (!a.ch_sigma || a.ch_causal) return cudaSuccess;
    const int64_t BH = (int64_t)a.B * a.H;
    LUNA_LAUNCH("chrms_scale", k_chrms_scale_rows, blocks_for(BH * a.D * a.dv), 256, 0, s, a.S_fin, a.z_fin,
                a.ch_sigma, BH, a.D, a.L, a.dv);
    return cudaGetLastError();
}

cudaError_t launch_chrms_dstate(const AttnArgs &a, cudaStream_t s) {
    if (!a.ch_sigma || a.ch_causal) return cudaSuccess;  // non-causal only, as above
    LUNA_LAUNCH("chrms_dstate", k_chrms_dstate, a.B * a.H, 128, 0, s, a, a.ch_sigma, a.ch_T);
    return cudaGetLastError();
}

cudaError_t launch_chrms_table(const AttnArgs &a, char *dst, cudaStream_t s) {
    LUNA_LAUNCH("chrms_table", k_chrms_scale_table, blocks_for(a.lay.bytes / 4), 256, 0, s,
                reinterpret_cast<const float *>(a.table), reinterpret_cast<float *>(dst), a.lay, a.ch_sigma);
    return cudaGetLastError();
}

cudaError_t launch_chrms_hist(const AttnArgs &a, cudaStream_t s) {
    if (!a.ch_sigma || !a.ch_causal) return cudaSuccess;
    LUNA_LAUNCH("chrms_hist", k_chrms_scale_hist, blocks_for((int64_t)a.lay.nint * a.lay.L * 2), 256, 0, s, a.hist,
                a.lay, a.ch_sigma);
    return cudaGetLastError();
}

cudaError_t launch_chrms_kappa(const AttnArgs &a, cudaStream_t s) {
    // non-causal: one T row per head; streaming form: one per block of the kernel that summed T
    const int trows = a.ch_causal ? a.ch_T_rows : a.B * a.H;
    LUNA_LAUNCH("chrms_kappa", k_chrms_kappa, 1, kRed, 0, s, a, a.ch_T, trows, a.ch_target, a.ch_stat,
                a.ch_causal ? a.ch_sigma : nullptr, a.ch_kappa);
    return cudaGetLastError();
}

bool tc_kterm_supported(const AttnArgs &a);
cudaError_t launch_tc_kterm(const AttnArgs &a, float *gpart, int max_parts, int *nparts, cudaStream_t s);

cudaError_t launch_chrms_backward(const AttnArgs &a, int main_parts, int *nparts, cudaStream_t s) {
    *nparts = main_parts;
    if (!a.ch_sigma) return cudaSuccess;
    cudaError_t e = launch_chrms_kappa(a, s);
    if (e != cudaSuccess) return e;
    if (tc_kterm_supported(a)) {  // the scale term on tensor cores (luna_tc_kterm.cu)
        int np = 0;
        if ((e = launch_tc_kterm(a, a.gpart + (size_t)main_parts * a.gsize, kChKBlocks, &np, s)) != cudaSuccess)
            return e;
        *nparts = main_parts + 2 * np;
        return cudaSuccess;
    }
    if (a.gpart64) {
        double *gpart = reinterpret_cast<double *>(a.gpart) + (size_t)main_parts * a.gsize;
        e = a.ch_io == LUNA_F32 ? kterm_impl<float>(a, gpart, s) : kterm_impl<__nv_bfloat16>(a, gpart, s);
    } else {
        float *gpart = a.gpart + (size_t)main_parts * a.gsize;
        e = a.ch_io == LUNA_F32 ? kterm_impl<float>(a, gpart, s) : kterm_impl<__nv_bfloat16>(a, gpart, s);
    }
    if (e != cudaSuccess) return e;
    *nparts = main_parts + 2 * kChKBlocks;
    return cudaSuccess;
}

}  // namespace luna
