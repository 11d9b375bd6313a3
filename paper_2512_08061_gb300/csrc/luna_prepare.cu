// Feature-map table: the exact piecewise-linear form of the channel MLPs.
//
// Each channel function of the listing's ScalarMLP is
//     psi_l(u) = relu( b2[l] + sum_k w2[l,k] relu(w1[l,k] u + b1[l,k]) ),
// a ReLU network of one scalar, hence linear in u between the kinks of its
// hidden units.  Merging the kinks of all L*hidden units into one sorted list
// T gives intervals j = #{p : T[p] < u} on which every hidden unit of every
// channel is either on or off, so
//     psi_l(u) = relu(alpha[j][l] * u + beta[j][l]).
// The kink of unit k is placed at the exact fp32 threshold of fma(w1, u, b1),
// so the interval reproduces the on/off decision of an fp32 evaluation of fc1
// for every fp32 u.  The 1/sqrt(M) scale of Eq. (phi-def-scalarenv) is folded
// into alpha and beta (it is positive, so relu commutes with it).
#include <math.h>

#include "luna_common.cuh"
#include "luna_prof.cuh"

namespace luna {

namespace {

__device__ float up_threshold(float w, float c) {
    // largest fp32 u with fma(w,u,c) <= 0, for w > 0 (fma is monotone in u)
    float t = -c / w;
    for (int it = 0; it < 64 && fmaf(w, t, c) > 0.0f; ++it) t = nextafterf(t, -INFINITY);
    for (int it = 0; it < 64 && fmaf(w, nextafterf(t, INFINITY), c) <= 0.0f; ++it) t = nextafterf(t, INFINITY);
    return t;
}

__device__ float down_threshold(float w, float c) {
    // largest fp32 u with fma(w,u,c) > 0, for w < 0
    float t = -c / w;
    for (int it = 0; it < 64 && !(fmaf(w, t, c) > 0.0f); ++it) t = nextafterf(t, -INFINITY);
    for (int it = 0; it < 64 && fmaf(w, nextafterf(t, INFINITY), c) > 0.0f; ++it) t = nextafterf(t, INFINITY);
    return t;
}

// Every block recomputes the thresholds and their ranks (512 x 512 compares)
// and then fills its slice of the (interval, channel) table; block 0 also
// writes the kink lists, the ranks and the parameter copies.  Per-unit values
// are kept in shared memory in [k][l] order, so that the eight channels read by
// a warp fall into eight consecutive banks.
constexpr int kPrepThreads = 256;

__global__ void __launch_bounds__(kPrepThreads) k_phi_prepare(luna_phi_params prm, TableLayout lay, char *table) {
    __shared__ float th[kMaxUnits];
    __shared__ int ty[kMaxUnits];
    __shared__ int rk[kMaxUnits];
    __shared__ float w1t[kMaxUnits], b1t[kMaxUnits], w2t[kMaxUnits];  // [k][l]
    __shared__ int tyt[kMaxUnits], rkt[kMaxUnits];                     // [k][l]
    __shared__ float srt[kMaxUnits];                                   // thresholds in sorted order
    const int tid = threadIdx.x, nt = blockDim.x;
    const int P = lay.P, L = lay.L, hid = lay.hid;

    for (int k = tid; k < P; k += nt) {
        const float w = prm.w1[k], c = prm.b1[k];
        if (w > 0.0f) { th[k] = up_threshold(w, c); ty[k] = 1; }
        else if (w < 0.0f) { th[k] = down_threshold(w, c); ty[k] = -1; }
        else { th[k] = INFINITY; ty[k] = (c > 0.0f) ? -1 : 1; }  // constant unit: always on / always off
    }
    __syncthreads();
    // rank by (threshold, unit index): a stable total order
    for (int k = tid; k < P; k += nt) {
        const float t = th[k];
        int r = 0;
        for (int q = 0; q < P; ++q) {
            const float sq = th[q];
            r += (sq < t || (sq == t && q < k)) ? 1 : 0;
        }
        rk[k] = r;
        srt[r] = t;
        const int l = k / hid, kk = k % hid, tpos = kk * L + l;
        w1t[tpos] = prm.w1[k]; b1t[tpos] = prm.b1[k]; w2t[tpos] = prm.w2[k];
        tyt[tpos] = ty[k]; rkt[tpos] = r;
    }
    __syncthreads();

    float *T = reinterpret_cast<float *>(table + lay.off_T);
    if (blockIdx.x == 0) {
        int *rank = reinterpret_cast<int *>(table + lay.off_rank);
        int *utype = reinterpret_cast<int *>(table + lay.off_utype);
        for (int k = tid; k < P; k += nt) {
            T[rk[k]] = th[k];
            rank[k] = rk[k];
            utype[k] = ty[k];
            reinterpret_cast<float *>(table + lay.off_w1)[k] = prm.w1[k];
            reinterpret_cast<float *>(table + lay.off_b1)[k] = prm.b1[k];
            reinterpret_cast<float *>(table + lay.off_w2)[k] = prm.w2[k];
        }
        for (int p = P + tid; p < lay.Ppad; p += nt) T[p] = INFINITY;
        // breadth-first (Eytzinger) copy: node e at depth d, position p in its
        // level holds the in-order element (2p+1) * 2^(9-d) - 1
        float *Te = reinterpret_cast<float *>(table + lay.off_Te);
        for (int e = tid; e < kEytzinger; e += nt) {
            float v = INFINITY;
            if (e > 0) {
                const int d = 31 - __clz(e);
                const int idx = ((2 * (e - (1 << d)) + 1) << (9 - d)) - 1;
                if (idx < P) v = srt[idx];
            }
            Te[e] = v;
        }
        float *W = reinterpret_cast<float *>(table + lay.off_W);
        for (int e = tid; e < lay.M * lay.d; e += nt) W[e] = prm.W[e];
        for (int e = tid; e < lay.M; e += nt) reinterpret_cast<float *>(table + lay.off_b)[e] = prm.b[e];
        for (int e = tid; e < L; e += nt) reinterpret_cast<float *>(table + lay.off_b2)[e] = prm.b2[e];
        if (tid == 0) {
            TableHeader *h = reinterpret_cast<TableHeader *>(table);
            h->magic = kTableMagic; h->version = kTableVersion;
            h->M = lay.M; h->L = lay.L; h->hid = lay.hid; h->d = lay.d; h->P = P; h->Ppad = lay.Ppad;
        }
    }
    // alpha, beta of every (interval j, channel l), scaled by 1/sqrt(M)
    float *AB = reinterpret_cast<float *>(table + lay.off_AB);
    const float scale = 1.0f / sqrtf((float)lay.M);
    for (int e = blockIdx.x * nt + tid; e < lay.nint * L; e += gridDim.x * nt) {
        const int j = e / L, l = e % L;
        float a = 0.0f, bsum = prm.b2[l];
        for (int k = 0; k < hid; ++k) {
            const int u = k * L + l;
            const bool on = (tyt[u] > 0) ? (rkt[u] < j) : (rkt[u] >= j);
            if (on) {
                a = fmaf(w2t[u], w1t[u], a);
                bsum = fmaf(w2t[u], b1t[u], bsum);
            }
        }
        AB[2 * e] = a * scale;
        AB[2 * e + 1] = bsum * scale;
    }
}

}  // namespace

cudaError_t launch_phi_prepare(const luna_phi_params &prm, const TableLayout &lay, void *table, cudaStream_t s) {
    const int blocks = (lay.nint * lay.L + kPrepThreads - 1) / kPrepThreads;
    LUNA_LAUNCH("phi_prepare", k_phi_prepare, blocks, kPrepThreads, 0, s, prm, lay, static_cast<char *>(table));
    return cudaGetLastError();
}

}  // namespace luna
