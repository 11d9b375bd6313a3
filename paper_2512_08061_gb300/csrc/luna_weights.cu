// Attention weights of a block of query rows, for the conversion's stage 1
// (appendix: the feature-map parameters are trained so that the attention
// distribution induced by the kernel matches the one of the original softmax
// module; the loss is not fixed by the paper, so the library only produces
// the two distributions).
//
//   LUNA (Eq. kernel-attn read as a weighted average of the values):
//       a_ij = k(q_i, k_j) / (sum_j' k(q_i, k_j') + eps),  k(x, y) = phi(x)^T phi(y)
//   teacher: p_ij = exp(q_i . k_j / sqrt(d)) / sum_j' exp(q_i . k_j' / sqrt(d))
//
// over the valid keys (j <= i in the streaming form); masked keys, query rows
// at or past the valid length and rows whose guarded sum is exactly 0 get 0.
// One block owns 32 query rows of one head and sweeps every key in tiles of
// 32 rows: pass 1 writes the raw scores (the kernel values, or the scaled dot
// products) and accumulates each row's sum (LUNA, in fp64) or its running
// maximum and rescaled exponential sum (teacher); pass 2 rereads the block's
// own rows and normalises them.  No scratch memory.
#include <math.h>

#include "luna_prof.cuh"
#include "luna_simt_dev.cuh"

namespace luna {
namespace {
using namespace simt;

constexpr int kWRows = 32;  // query rows per block
constexpr int kWKeys = 32;  // key rows per tile
constexpr int kWLanes = kThreads / kWRows;  // threads per query row (8): keys jj, jj + 8, ...

template <typename IO>
__global__ void __launch_bounds__(kThreads) k_weights(AttnArgs a, int causal, int row0, int rows, int teacher, int64_t tstride,
                                                                float *A) {
    extern __shared__ __align__(16) float smem[];
    Carve cv{smem};
    const TableLayout &lay = a.lay;
    const int D = a.D, d = a.d, n = a.n;
    SmemPhi s = carve_phi(cv, lay);
    float *sQ = cv.take(kWRows * d);
    float *sPq = cv.take(kWRows * D);
    float *sK = cv.take(kWKeys * d);
    float *sPk = cv.take(kWKeys * D);
    if (!carve_fits(cv, smem)) return;
    const int bh = blockIdx.y;
    const int len = head_length(a.lengths, bh / a.H, n);
    const int r_lo = blockIdx.x * kWRows;              // first output row of this block (relative to row0)
    const int nr = min(kWRows, rows - r_lo);           // output rows of this block
    const int i_lo = row0 + r_lo;                      // its first query row
    const int nq = max(0, min(nr, len - i_lo));        // of which valid query rows
    float *Ab = A + ((size_t)bh * rows + r_lo) * n;
    const IO *Qh = static_cast<const IO *>(a.Q) + (size_t)bh * n * d;
    const IO *Kh = static_cast<const IO *>(a.K) + (size_t)bh * n * d;
    // rows past the valid length: zeros
    for (size_t e = (size_t)nq * n + threadIdx.x; e < (size_t)nr * n; e += blockDim.x) Ab[e] = 0.0f;
    if (nq == 0) return;
    if (!teacher) load_phi(s, lay, a.table + (size_t)(bh % a.H) * tstride);  // this head's table
    load_rows(sQ, Qh + (size_t)i_lo * d, nq * d);
    __syncthreads();
    if (!teacher) phi_tile(lay, s, sQ, nq, sPq, nullptr, nullptr);
    const int r = threadIdx.x / kWLanes, jj = threadIdx.x % kWLanes;
    const int i = i_lo + r;
    const bool rv = r < nq;
    const int jmax = !rv ? 0 : (causal ? min(i + 1, len) : len);  // keys this row sees
    const int jend = causal ? min(i_lo + nq, len) : len;           // keys the block needs
    const float qscale = 1.0f / sqrtf((float)d);
    double lsum = 0.0;                                 // LUNA: row sum of the kernel values
    float mx = -INFINITY, esum = 0.0f;                 // teacher: running maximum and exponential sum
    float *Ar = Ab + (size_t)r * n;
    for (int j0 = 0; j0 < n; j0 += kWKeys) {
        const int nk = min(kWKeys, n - j0);
        if (j0 < jend) {
            __syncthreads();
            load_rows(sK, Kh + (size_t)j0 * d, min(nk, jend - j0) * d);
            __syncthreads();
            if (!teacher) {
                phi_tile(lay, s, sK, min(nk, jend - j0), sPk, nullptr, nullptr);
                __syncthreads();
            }
        }
        if (!rv) continue;
        for (int t = jj; t < nk; t += kWLanes) {
            const int j = j0 + t;
            float v = 0.0f;
            if (j < jmax) {
                float acc = 0.0f;
                if (teacher) {
                    for (int c = 0; c < d; ++c) acc = fmaf(sQ[r * d + c], sK[t * d + c], acc);
                    acc *= qscale;
                    if (acc > mx) {
                        esum *= expf(mx - acc);
                        mx = acc;
                    }
                    esum += expf(acc - mx);
                } else {
                    for (int f = 0; f < D; ++f) acc = fmaf(sPq[r * D + f], sPk[t * D + f], acc);
                    lsum += (double)acc;
                }
                v = acc;
            }
            Ar[j] = (j < jmax) ? v : 0.0f;
        }
    }
    // combine the row's lanes (kWLanes consecutive threads of one warp)
    float scale = 0.0f;
    if (teacher) {
#pragma unroll
        for (int o = kWLanes / 2; o > 0; o >>= 1) {
            const float m2 = __shfl_xor_sync(0xffffffffu, mx, o), e2 = __shfl_xor_sync(0xffffffffu, esum, o);
            const float m = fmaxf(mx, m2);
            esum = (m == -INFINITY) ? 0.0f : esum * expf(mx - m) + e2 * expf(m2 - m);
            mx = m;
        }
        scale = esum > 0.0f ? 1.0f / esum : 0.0f;
    } else {
#pragma unroll
        for (int o = kWLanes / 2; o > 0; o >>= 1) lsum += __shfl_xor_sync(0xffffffffu, lsum, o);
        const double den = lsum + (double)a.eps;
        scale = den != 0.0 ? (float)(1.0 / den) : 0.0f;
    }
    __syncthreads();
    if (!rv) return;
    // pass 2: normalise the row (this thread's own entries, written above)
    for (int j = jj; j < jmax; j += kWLanes) {
        const float v = Ar[j];
        Ar[j] = teacher ? expf(v - mx) * scale : v * scale;
    }
}

size_t smem_weights(const AttnArgs &a) {
    HostCarve cv;
    carve_phi_host(cv, a.lay);
    cv.take(kWRows * a.d); cv.take(kWRows * a.D); cv.take(kWKeys * a.d); cv.take(kWKeys * a.D);
    return cv.bytes();
}

template <typename IO>
cudaError_t weights_impl(const AttnArgs &a, int causal, int row0, int rows, int teacher, int64_t tstride, float *A,
                         cudaStream_t s) {
    const size_t sm = smem_weights(a);
    cudaError_t e = set_smem(k_weights<IO>, sm);
    if (e != cudaSuccess) return e;
    const dim3 grid((rows + kWRows - 1) / kWRows, a.B * a.H);
    LUNA_LAUNCH("weights", k_weights<IO>, grid, kThreads, sm, s, a, causal, row0, rows, teacher, tstride, A);
    return cudaGetLastError();
}

}  // namespace

size_t weights_max_smem(const AttnArgs &a) { return smem_weights(a); }

cudaError_t launch_weights(const AttnArgs &a, luna_dtype io, int causal, int row0, int rows, int teacher,
                           int64_t tstride, float *A, cudaStream_t s) {
    return io == LUNA_F32 ? weights_impl<float>(a, causal, row0, rows, teacher, tstride, A, s)
                          : weights_impl<__nv_bfloat16>(a, causal, row0, rows, teacher, tstride, A, s);
}

}  // namespace luna
