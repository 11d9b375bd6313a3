// Device helpers shared by the CUDA-core kernels (non-causal and causal).
#pragma once

#include "luna_simt.cuh"

namespace luna {
namespace simt {
namespace {  // internal linkage in every translation unit that includes this

constexpr int kThreads = 256;
constexpr int kTileK = 32;  // rows per tile, key statistics
constexpr int kTileQ = 32;  // rows per block, query pass
constexpr int kTileB = 16;  // rows per tile, backward passes
constexpr int kPhiRows = 32;  // rows of one phi_tile / phi_backward_tile call at most (the variants' row scratch)

__host__ __device__ inline int r4(int x) { return (x + 3) & ~3; }

struct Carve {
    float *p;
    __device__ float *take(int n) {
        float *r = p;
        p += r4(n);
        return r;
    }
};

// True when the arrays carved so far fit in the block's dynamic shared memory (the host sizes the
// launch with a HostCarve of the same arrays; a kernel whose carve does not fit returns before it
// touches shared memory, so a mismatch shows as a wrong result, not as an out-of-bounds access).
__device__ __forceinline__ bool carve_fits(const Carve &cv, const float *base) {
    uint32_t dyn;
    asm volatile("mov.u32 %0, %%dynamic_smem_size;" : "=r"(dyn));
    return (size_t)(cv.p - base) * sizeof(float) <= (size_t)dyn;
}

struct HostCarve {
    int n = 0;
    void take(int k) { n += r4(k); }
    size_t bytes() const { return (size_t)n * 4; }
};

// The feature map in shared memory: the sorted kinks T and the interval table AB (ReLU MLPs), or the
// MLP parameters themselves (another activation: direct evaluation); the projection; the variants'
// gate and coefficients with their per-row scratch.
struct SmemPhi {
    float *T, *AB, *W, *b;
    float *w1, *b1, *w2, *b2;  // channel MLPs (non-ReLU activation)
    float *We, *be, *coef;     // envelope gate, Bank+Coef coefficients
    float *E, *H, *dE;         // [kPhiRows][L] per row: e_l = h_l c_l, the gate h_l, dLoss/de_l (then the gate's
                               // pre-activation gradient)
};

__device__ SmemPhi carve_phi(Carve &cv, const TableLayout &lay) {
    SmemPhi s = {};
    if (!lay.act) {
        s.T = cv.take(lay.Ppad);
        s.AB = cv.take(lay.nint * ab_stride(lay));
    }
    s.W = cv.take(lay.M * lay.d);
    s.b = cv.take(lay.M);
    if (lay.act) {
        s.w1 = cv.take(lay.P); s.b1 = cv.take(lay.P); s.w2 = cv.take(lay.L * lay.hid); s.b2 = cv.take(lay.L);
    }
    if (lay.env) { s.We = cv.take(lay.L * lay.d); s.be = cv.take(lay.L); }
    if (lay.coef) s.coef = cv.take(lay.L);
    if (lay.env || lay.coef) {
        s.E = cv.take(kPhiRows * lay.L); s.H = cv.take(kPhiRows * lay.L); s.dE = cv.take(kPhiRows * lay.L);
    }
    return s;
}
void carve_phi_host(HostCarve &cv, const TableLayout &lay) {
    if (!lay.act) { cv.take(lay.Ppad); cv.take(lay.nint * ab_stride(lay)); }
    cv.take(lay.M * lay.d); cv.take(lay.M);
    if (lay.act) { cv.take(lay.P); cv.take(lay.P); cv.take(lay.L * lay.hid); cv.take(lay.L); }
    if (lay.env) { cv.take(lay.L * lay.d); cv.take(lay.L); }
    if (lay.coef) cv.take(lay.L);
    if (lay.env || lay.coef) { cv.take(kPhiRows * lay.L); cv.take(kPhiRows * lay.L); cv.take(kPhiRows * lay.L); }
}

// The (alpha, beta) table into shared memory at ab_stride(lay) words per interval.
__device__ void copy_ab(float *dst, const TableLayout &lay, const char *table) {
    const float *src = reinterpret_cast<const float *>(table + lay.off_AB);
    const int w = 2 * lay.L, st = ab_stride(lay);
    for (int e = threadIdx.x; e < lay.nint * w; e += blockDim.x) dst[(e / w) * st + e % w] = src[e];
}

// (alpha, beta) of channel l in the entry of one interval.
__device__ __forceinline__ float2 ab_pair(const float *entry, int l) { return reinterpret_cast<const float2 *>(entry)[l]; }

__device__ void load_phi(const SmemPhi &s, const TableLayout &lay, const char *table) {
    auto copy = [&](float *dst, int64_t off, int count) {
        const float *src = reinterpret_cast<const float *>(table + off);
        for (int e = threadIdx.x; e < count; e += blockDim.x) dst[e] = src[e];
    };
    if (!lay.act) {
        copy(s.T, lay.off_T, lay.Ppad);
        copy_ab(s.AB, lay, table);
    }
    copy(s.W, lay.off_W, lay.M * lay.d);
    copy(s.b, lay.off_b, lay.M);
    if (lay.act) {
        copy(s.w1, lay.off_w1, lay.P); copy(s.b1, lay.off_b1, lay.P);
        copy(s.w2, lay.off_w2, lay.L * lay.hid); copy(s.b2, lay.off_b2, lay.L);
    }
    if (lay.env) { copy(s.We, lay.off_We, lay.L * lay.d); copy(s.be, lay.off_be, lay.L); }
    if (lay.coef) copy(s.coef, lay.off_coef, lay.L);
}

// The channel MLPs' hidden activation (luna_act) and its derivative da (ReLU'(0) = 0).
// GELU(a) = a Phi(a), Phi(a) = (1 + erf(a / sqrt 2)) / 2, GELU' = Phi(a) + a exp(-a^2 / 2) / sqrt(2 pi);
// SiLU(a) = a sigma(a), SiLU' = sigma (1 + a (1 - sigma)); tanh' = 1 - tanh^2.
__device__ __forceinline__ float act_eval(int act, float a, float &da) {
    switch (act) {
        case LUNA_ACT_GELU: {
            const float c = 0.5f * (1.0f + erff(a * 0.70710678118654752f));
            da = fmaf(a * 0.39894228040143268f, expf(-0.5f * a * a), c);
            return a * c;
        }
        case LUNA_ACT_SILU: {
            const float sg = 1.0f / (1.0f + expf(-a));
            da = sg * fmaf(a, 1.0f - sg, 1.0f);
            return a * sg;
        }
        case LUNA_ACT_TANH: {
            const float t = tanhf(a);
            da = fmaf(-t, t, 1.0f);
            return t;
        }
        default:
            da = a > 0.0f ? 1.0f : 0.0f;
            return fmaxf(a, 0.0f);
    }
}

// The 1/sqrt(M) of Eq. (phi-def-scalarenv), as the table folds it into alpha and beta.
__device__ __forceinline__ float phi_scale(const TableLayout &lay) { return 1.0f / sqrtf((float)lay.M); }

// Direct evaluation of channel l's MLP output y_l(u) = b2_l + sum_k w2_lk act(w1 u + b1) (before the outer
// ReLU and the scale); with dydu, also dy/du = sum_k w2_lk act'(w1 u + b1) w1.
__device__ __forceinline__ float channel_direct(const TableLayout &lay, const SmemPhi &s, int l, float u,
                                                float *dydu) {
    const int hid = lay.hid, base = lay.shared ? 0 : l * hid;
    const float *w2 = s.w2 + l * hid;
    float y = s.b2[l], t = 0.0f;
    for (int k = 0; k < hid; ++k) {
        float da;
        const float w1 = s.w1[base + k];
        const float av = act_eval(lay.act, fmaf(w1, u, s.b1[base + k]), da);
        y = fmaf(w2[k], av, y);
        t = fmaf(w2[k] * da, w1, t);
    }
    if (dydu) *dydu = t;
    return y;
}

// The ungated channel value phi0 = max(scale y_l(u), floor) of interval j (table) or by direct evaluation.
__device__ __forceinline__ float channel_value(const TableLayout &lay, const SmemPhi &s, float u, int j, int l,
                                               float fl) {
    if (lay.act) return fmaxf(phi_scale(lay) * channel_direct(lay, s, l, u, nullptr), fl);
    const float2 ab = ab_pair(s.AB + j * ab_stride(lay), l);
    return fmaxf(fmaf(ab.x, u, ab.y), fl);
}

// Per-row factors of the variants for rows [0, nr) of sX: H = h_l(x) = sigmoid(We_l . x + be_l) (1 without the
// gate), E = h_l c_l (c_l = 1 without Bank+Coef).
__device__ void gate_rows(const TableLayout &lay, const SmemPhi &s, const float *sX, int nr) {
    const int L = lay.L, d = lay.d;
    for (int e = threadIdx.x; e < nr * L; e += blockDim.x) {
        const int r = e / L, l = e - r * L;
        float h = 1.0f;
        if (lay.env) {
            float a = s.be[l];
            for (int c = 0; c < d; ++c) a = fmaf(s.We[l * d + c], sX[r * d + c], a);
            h = 1.0f / (1.0f + expf(-a));
        }
        s.H[e] = h;
        s.E[e] = lay.coef ? h * s.coef[l] : h;
    }
}

template <typename IO>
__device__ void load_rows(float *dst, const IO *src, int count) {
    for (int e = threadIdx.x; e < count; e += blockDim.x) dst[e] = io_load(src + e);
}

// phi for rows [0, nr) of a row tile sX (row stride d) into sPhi (row stride D).
// Optionally keeps the projections u and their merged interval j (0 with direct evaluation).
// Called by every thread of the block; with a gate or coefficients it synchronises the block.
__device__ void phi_tile(const TableLayout &lay, const SmemPhi &s, const float *sX, int nr, float *sPhi, float *sU,
                         int *sJ) {
    const int M = lay.M, L = lay.L, d = lay.d, D = lay.D;
    const float fl = channel_floor(lay);
    const bool ev = lay.env || lay.coef;
    if (ev) {
        __syncthreads();  // the row scratch of an earlier call is no longer read
        gate_rows(lay, s, sX, nr);
        __syncthreads();
    }
    const float sc = phi_scale(lay);
    for (int e = threadIdx.x; e < nr * M; e += blockDim.x) {
        const int r = e / M, i = e - r * M;
        const float *x = sX + r * d;
        const float *w = s.W + i * d;
        float u = s.b[i];
        for (int c = 0; c < d; ++c) u = fmaf(w[c], x[c], u);
        float *out = sPhi + r * D + i * L;
        int j = 0;
        if (!lay.act) {
            j = interval_of(s.T, lay.Ppad, u);
            const float *ab = s.AB + j * ab_stride(lay);
            for (int l = 0; l < L; ++l) {
                const float2 p = ab_pair(ab, l);
                out[l] = fmaxf(fmaf(p.x, u, p.y), fl);
            }
        } else {
            for (int l = 0; l < L; ++l) out[l] = fmaxf(sc * channel_direct(lay, s, l, u, nullptr), fl);
        }
        if (ev)
            for (int l = 0; l < L; ++l) out[l] *= s.E[r * L + l];
        if (sU) { sU[e] = u; sJ[e] = j; }
    }
}

// acc[k][m] += sum_r A[r][f0+k] * Bm[r][c0+m];  z[k] += sum_r A[r][f0+k] * (w ? w[r] : 1), accumulated in fp64:
// the statistics (S, z and dS, dz) are sums over every row of a head, and their rounding is shared by every
// row that reads them, so it does not average out in the parameter gradients
__device__ __forceinline__ void outer_accumulate(double (&acc)[8][8], double (&zacc)[8], bool do_z, const float *sA,
                                                 int D, const float *sB, int dv, const float *sw, int nr, int f0,
                                                 int c0) {
    for (int r = 0; r < nr; ++r) {
        double a8[8], b8[8];
#pragma unroll
        for (int k = 0; k < 8; ++k) {
            a8[k] = (f0 + k < D) ? (double)sA[r * D + f0 + k] : 0.0;
            b8[k] = (c0 + k < dv) ? (double)sB[r * dv + c0 + k] : 0.0;
        }
#pragma unroll
        for (int k = 0; k < 8; ++k)
#pragma unroll
            for (int m = 0; m < 8; ++m) acc[k][m] = fma(a8[k], b8[m], acc[k][m]);
        if (do_z) {
            const double wr = sw ? (double)sw[r] : 1.0;
#pragma unroll
            for (int k = 0; k < 8; ++k) zacc[k] = fma(a8[k], wr, zacc[k]);
        }
    }
}

__device__ bool last_arrival(int *counter, int expected) {
    __shared__ int s_flag;
    __threadfence();
    __syncthreads();
    if (threadIdx.x == 0) s_flag = (atomicAdd(counter, 1) == expected - 1) ? 1 : 0;
    __syncthreads();
    if (s_flag) __threadfence();
    return s_flag != 0;
}

// out[e] = sum_p part[p][e] in order p = 0..nparts-1 (fp64, rounded once)
__device__ void ordered_sum(const float *part, int nparts, int count, float *out) {
    for (int e = threadIdx.x; e < count; e += blockDim.x) {
        double s = 0.0;
        for (int p0 = 0; p0 < nparts; p0 += 8) {  // eight loads in flight, added in order
            float v[8];
#pragma unroll
            for (int k = 0; k < 8; ++k) v[k] = (p0 + k < nparts) ? __ldcg(part + (size_t)(p0 + k) * count + e) : 0.0f;
#pragma unroll
            for (int k = 0; k < 8; ++k)
                if (p0 + k < nparts) s += (double)v[k];
        }
        out[e] = (float)s;
    }
}

// Exclusive scan over partials in order: forward (out[p] = sum_{q<p} part[q],
// out[nparts] = total) or reverse (out[p] = sum_{q>p} part[q]); fp64 running sums, each output rounded once.
__device__ void exclusive_scan(const float *part, int nparts, int count, float *out, bool reverse) {
    for (int e = threadIdx.x; e < count; e += blockDim.x) {
        double s = 0.0;
        if (!reverse) {
            for (int p = 0; p < nparts; ++p) {
                out[(size_t)p * count + e] = (float)s;
                s += (double)__ldcg(part + (size_t)p * count + e);
            }
            out[(size_t)nparts * count + e] = (float)s;
        } else {
            for (int p = nparts - 1; p >= 0; --p) {
                out[(size_t)p * count + e] = (float)s;
                s += (double)__ldcg(part + (size_t)p * count + e);
            }
        }
    }
}

// Writes a (D x dv) register-tiled accumulator and its z-vector to a partial slot.
__device__ void store_tile(const double (&acc)[8][8], const double (&zacc)[8], bool active, int tc, int f0, int c0,
                           int D, int dv, float *Sp, float *zp) {
    if (!active) return;
#pragma unroll
    for (int k = 0; k < 8; ++k)
#pragma unroll
        for (int m = 0; m < 8; ++m)
            if (f0 + k < D && c0 + m < dv) Sp[(f0 + k) * dv + c0 + m] = acc[k][m];
    if (tc == 0)
#pragma unroll
        for (int k = 0; k < 8; ++k)
            if (f0 + k < D) zp[f0 + k] = zacc[k];
}

// ---------------------------------------------------------------------------
// backward through phi for a tile: dU = sum_l dPhi * dphi/du, histogram of
// the channel-MLP gradient statistics, then dX = dU W and dW += dU^T X.

// The parameter gradients are sums over every row, projection and channel whose terms cancel (the
// loss is nearly invariant to a common scale of the features), so the generic kernels accumulate them,
// and the histogram, in fp64; the per-sample terms stay fp32.
struct GradAcc {
    double dW[16];  // entries threadIdx.x + k * blockDim.x of the M*d matrix
    double db;      // entry threadIdx.x of b (if < M)
};

__device__ void phi_backward_tile(const TableLayout &lay, const SmemPhi &s, const float *sX, int nr,
                                  const float *sPhi, float *sdPhi, const float *sU, const int *sJ, float *sdU,
                                  double *shist, double *gvar, GradAcc &g) {
    const int M = lay.M, L = lay.L, d = lay.d, D = lay.D;
    const float fl = channel_floor(lay);
    const bool ev = lay.env || lay.coef;
    const float sc = phi_scale(lay);
    if (ev) {
        // phi = e_l phi0 with e_l = h_l(x) c_l per row: dLoss/de_l = sum over the projections of dPhi phi0
        __syncthreads();  // the row scratch of an earlier call is no longer read
        gate_rows(lay, s, sX, nr);
        for (int e = threadIdx.x; e < nr * L; e += blockDim.x) {
            const int r = e / L, l = e - r * L;
            double acc = 0.0;
            for (int i = 0; i < M; ++i)
                acc = fma((double)sdPhi[r * D + i * L + l],
                          (double)channel_value(lay, s, sU[r * M + i], sJ[r * M + i], l, fl), acc);
            s.dE[e] = (float)acc;
        }
        __syncthreads();
    }
    // per sample (row, projection): g_l = dLoss/dphi0_l on an active output; dU = sum_l g_l dphi0_l/du
    for (int e = threadIdx.x; e < nr * M; e += blockDim.x) {
        const int r = e / M, i = e - r * M;
        const float u = sU[e];
        double du = 0.0;
        if (!lay.act) {
            const int j = sJ[e];
            const float *ab = s.AB + j * ab_stride(lay);
            for (int l = 0; l < L; ++l) {
                const int f = r * D + i * L + l;
                const float2 p = ab_pair(ab, l);
                const bool on = ev ? fmaf(p.x, u, p.y) > fl : sPhi[f] > fl;
                if (on) {  // outer ReLU on (always, for signed outputs)
                    const double gl = ev ? (double)sdPhi[f] * (double)s.E[r * L + l] : (double)sdPhi[f];
                    du = fma(gl, (double)p.x, du);
                    if (gl != 0.0) {
                        atomicAdd(shist + (j * L + l) * 2, gl);
                        atomicAdd(shist + (j * L + l) * 2 + 1, gl * (double)u);  // exact product
                    }
                }
            }
        } else {
            // direct evaluation: G_l = dLoss/dy_l (scale and gate folded in), kept in sdPhi for the unit sums
            for (int l = 0; l < L; ++l) {
                const int f = r * D + i * L + l;
                float dydu;
                const float y = channel_direct(lay, s, l, u, &dydu);
                float G = 0.0f;
                if (sc * y > fl) G = (ev ? sdPhi[f] * s.E[r * L + l] : sdPhi[f]) * sc;
                du = fma((double)G, (double)dydu, du);
                sdPhi[f] = G;
            }
        }
        sdU[e] = (float)du;
    }
    __syncthreads();
    if (lay.act) {
        // MLP gradients unit by unit over the tile's samples, into the block's partial
        // [dw2 (L*hid) | dw1 (P) | db1 (P) | db2 (L)]; each entry has one owner thread
        const int hid = lay.hid, P = lay.P, ns = nr * M;
        double *dw2 = shist, *dw1 = shist + L * hid, *db1 = dw1 + P, *db2 = db1 + P;
        if (!lay.shared) {
            for (int q = threadIdx.x; q < P; q += blockDim.x) {
                const int l = q / hid;
                const float w1 = s.w1[q], b1 = s.b1[q], w2 = s.w2[q];
                double a2 = 0.0, a1 = 0.0, a0 = 0.0;
                for (int e = 0; e < ns; ++e) {
                    const int r = e / M, i = e - r * M;
                    const float G = sdPhi[r * D + i * L + l];
                    if (G == 0.0f) continue;
                    float da;
                    const float av = act_eval(lay.act, fmaf(w1, sU[e], b1), da);
                    a2 = fma((double)G, (double)av, a2);
                    const double dh = (double)G * (double)w2 * (double)da;
                    a0 += dh;
                    a1 = fma(dh, (double)sU[e], a1);
                }
                dw2[q] += a2; dw1[q] += a1; db1[q] += a0;
            }
        } else {
            for (int k = threadIdx.x; k < hid; k += blockDim.x) {
                const float w1 = s.w1[k], b1 = s.b1[k];
                double a2[kMaxL] = {}, a1 = 0.0, a0 = 0.0;
                for (int e = 0; e < ns; ++e) {
                    const int r = e / M, i = e - r * M;
                    float da;
                    const float av = act_eval(lay.act, fmaf(w1, sU[e], b1), da);
                    double dsum = 0.0;  // sum over the channels of G_l w2_lk
                    for (int l = 0; l < L; ++l) {
                        const float G = sdPhi[r * D + i * L + l];
                        a2[l] = fma((double)G, (double)av, a2[l]);
                        dsum = fma((double)G, (double)s.w2[l * hid + k], dsum);
                    }
                    const double dh = dsum * (double)da;
                    a0 += dh;
                    a1 = fma(dh, (double)sU[e], a1);
                }
                for (int l = 0; l < L; ++l) dw2[l * hid + k] += a2[l];
                dw1[k] += a1; db1[k] += a0;
            }
        }
        for (int l = threadIdx.x; l < L; l += blockDim.x) {
            double acc = 0.0;
            for (int e = 0; e < ns; ++e) acc += (double)sdPhi[(e / M) * D + (e % M) * L + l];
            db2[l] += acc;
        }
    }
    if (ev) {
        // Bank+Coef: dc_l = sum over rows of dLoss/de_l h_l; the gate: dLoss/d(We_l . x + be_l) = dLoss/de_l c_l h (1 - h)
        // (kept in dE for store_dx's dX term), then dWe = sum_r that x_r^T and dbe = sum_r that
        double *dWe = gvar, *dbe = gvar + L * d, *dcoef = gvar + (lay.env ? L * d + L : 0);
        if (lay.coef)
            for (int l = threadIdx.x; l < L; l += blockDim.x) {
                double acc = 0.0;
                for (int r = 0; r < nr; ++r) acc = fma((double)s.dE[r * L + l], (double)s.H[r * L + l], acc);
                dcoef[l] += acc;
            }
        if (lay.env) {
            __syncthreads();  // dE read above
            for (int e = threadIdx.x; e < nr * L; e += blockDim.x) {
                const float h = s.H[e], c = lay.coef ? s.coef[e % L] : 1.0f;
                s.dE[e] = s.dE[e] * c * h * (1.0f - h);
            }
            __syncthreads();
            for (int q = threadIdx.x; q < L * d; q += blockDim.x) {
                const int l = q / d, c = q - l * d;
                double acc = 0.0;
                for (int r = 0; r < nr; ++r) acc = fma((double)s.dE[r * L + l], (double)sX[r * d + c], acc);
                dWe[q] += acc;
            }
            for (int l = threadIdx.x; l < L; l += blockDim.x) {
                double acc = 0.0;
                for (int r = 0; r < nr; ++r) acc += (double)s.dE[r * L + l];
                dbe[l] += acc;
            }
        }
    }
    for (int k = 0; k < 16; ++k) {
        const int e = threadIdx.x + k * blockDim.x;
        if (e >= M * d) break;
        const int i = e / d, c = e - i * d;
        double acc = g.dW[k];
        for (int r = 0; r < nr; ++r) acc = fma((double)sdU[r * M + i], (double)sX[r * d + c], acc);
        g.dW[k] = acc;
    }
    if (threadIdx.x < M)
        for (int r = 0; r < nr; ++r) g.db += (double)sdU[r * M + threadIdx.x];
}

// dX = dU W (+ the envelope gate's term sum_l dLoss/d(We_l . x + be_l) We_l, kept in dE by phi_backward_tile).
template <typename IO>
__device__ void store_dx(const TableLayout &lay, const SmemPhi &s, const float *sdU, int nr, IO *dX) {
    const int M = lay.M, d = lay.d, L = lay.L;
    for (int e = threadIdx.x; e < nr * d; e += blockDim.x) {
        const int r = e / d, c = e - r * d;
        float acc = 0.0f;
        for (int i = 0; i < M; ++i) acc = fmaf(sdU[r * M + i], s.W[i * d + c], acc);
        if (lay.env)
            for (int l = 0; l < L; ++l) acc = fmaf(s.dE[r * L + l], s.We[l * d + c], acc);
        io_store(dX + e, acc);
    }
}

// Writes dW and db into the block's fp64 partial gp = [dW | db | histogram]; the histogram was
// accumulated in place.
__device__ void store_grad_partial(const TableLayout &lay, const GradAcc &g, double *gp) {
    const int Md = lay.M * lay.d;
    for (int k = 0; k < 16; ++k) {
        const int e = threadIdx.x + k * blockDim.x;
        if (e >= Md) break;
        gp[e] = g.dW[k];
    }
    if (threadIdx.x < lay.M) gp[Md + threadIdx.x] = g.db;
}

template <typename K>
cudaError_t set_smem(K kernel, size_t bytes) {
    return cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)bytes);
}


}  // namespace
}  // namespace simt
}  // namespace luna
