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

struct SmemPhi {
    float *T, *AB, *W, *b;
};

__device__ SmemPhi carve_phi(Carve &cv, const TableLayout &lay) {
    SmemPhi s;
    s.T = cv.take(lay.Ppad);
    s.AB = cv.take(lay.nint * lay.L * 2);
    s.W = cv.take(lay.M * lay.d);
    s.b = cv.take(lay.M);
    return s;
}
void carve_phi_host(HostCarve &cv, const TableLayout &lay) {
    cv.take(lay.Ppad); cv.take(lay.nint * lay.L * 2); cv.take(lay.M * lay.d); cv.take(lay.M);
}

__device__ void load_phi(const SmemPhi &s, const TableLayout &lay, const char *table) {
    const float *T = reinterpret_cast<const float *>(table + lay.off_T);
    const float *AB = reinterpret_cast<const float *>(table + lay.off_AB);
    const float *W = reinterpret_cast<const float *>(table + lay.off_W);
    const float *b = reinterpret_cast<const float *>(table + lay.off_b);
    for (int e = threadIdx.x; e < lay.Ppad; e += blockDim.x) s.T[e] = T[e];
    for (int e = threadIdx.x; e < lay.nint * lay.L * 2; e += blockDim.x) s.AB[e] = AB[e];
    for (int e = threadIdx.x; e < lay.M * lay.d; e += blockDim.x) s.W[e] = W[e];
    for (int e = threadIdx.x; e < lay.M; e += blockDim.x) s.b[e] = b[e];
}

template <typename IO>
__device__ void load_rows(float *dst, const IO *src, int count) {
    for (int e = threadIdx.x; e < count; e += blockDim.x) dst[e] = io_load(src + e);
}

// phi for rows [0, nr) of a row tile sX (row stride d) into sPhi (row stride D).
// Optionally keeps the projections u and their merged interval j.
__device__ void phi_tile(const TableLayout &lay, const SmemPhi &s, const float *sX, int nr, float *sPhi, float *sU,
                         int *sJ) {
    const int M = lay.M, L = lay.L, d = lay.d, D = lay.D;
    const float fl = channel_floor(lay);
    for (int e = threadIdx.x; e < nr * M; e += blockDim.x) {
        const int r = e / M, i = e - r * M;
        const float *x = sX + r * d;
        const float *w = s.W + i * d;
        float u = s.b[i];
        for (int c = 0; c < d; ++c) u = fmaf(w[c], x[c], u);
        const int j = interval_of(s.T, lay.Ppad, u);
        const float *ab = s.AB + j * L * 2;
        float *out = sPhi + r * D + i * L;
        for (int l = 0; l < L; ++l) out[l] = fmaxf(fmaf(ab[2 * l], u, ab[2 * l + 1]), fl);
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
                                  const float *sPhi, const float *sdPhi, const float *sU, const int *sJ, float *sdU,
                                  double *shist, GradAcc &g) {
    const int M = lay.M, L = lay.L, d = lay.d, D = lay.D;
    const float fl = channel_floor(lay);
    for (int e = threadIdx.x; e < nr * M; e += blockDim.x) {
        const int r = e / M, i = e - r * M;
        const float u = sU[e];
        const int j = sJ[e];
        const float *ab = s.AB + j * L * 2;
        double du = 0.0;
        for (int l = 0; l < L; ++l) {
            const int f = r * D + i * L + l;
            if (sPhi[f] > fl) {  // outer ReLU on (always, for signed outputs)
                const double gl = sdPhi[f];
                du = fma(gl, (double)ab[2 * l], du);
                if (gl != 0.0) {
                    atomicAdd(shist + (j * L + l) * 2, gl);
                    atomicAdd(shist + (j * L + l) * 2 + 1, gl * (double)u);  // exact product
                }
            }
        }
        sdU[e] = (float)du;
    }
    __syncthreads();
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

template <typename IO>
__device__ void store_dx(const TableLayout &lay, const SmemPhi &s, const float *sdU, int nr, IO *dX) {
    const int M = lay.M, d = lay.d;
    for (int e = threadIdx.x; e < nr * d; e += blockDim.x) {
        const int r = e / d, c = e - r * d;
        float acc = 0.0f;
        for (int i = 0; i < M; ++i) acc = fmaf(sdU[r * M + i], s.W[i * d + c], acc);
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
