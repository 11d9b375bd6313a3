// Feature-map table: the exact piecewise-linear form of the channel MLPs.
//
// Each channel function of the listing's ScalarMLP is
//     psi_l(u) = relu( b2[l] + sum_k w2[l,k] relu(w1[l,k] u + b1[l,k]) )
// (with the shared-channel MLP, w1[k], b1[k] for every l), a ReLU network of
// one scalar, hence linear in u between the kinks of its hidden units.
// Merging the kinks of all P hidden units (L*hidden, or hidden when shared)
// into one sorted list
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

// One launch: every block computes the kink threshold of every hidden unit and
// sorts the (threshold, unit index) pairs (a bitonic network over one element
// per thread: warp shuffles for partners within a warp, shared memory across
// warps; a stable total order), then computes its slice of alpha and beta,
// eight threads per (interval, channel) entry; block 0 also writes the sorted
// kink list and interval search block, each unit's rank and active side, and the
// parameter copies.
constexpr int kPrepThreads = kMaxUnits;                       // one thread per (padded) unit
constexpr int kPrepSplit = 8;                                 // threads per (interval, channel) entry
constexpr int kPrepEntries = kPrepThreads / kPrepSplit;       // entries per block

__device__ __forceinline__ bool pair_less(float ta, int ka, float tb, int kb) {
    return ta < tb || (ta == tb && ka < kb);
}

// Bitonic sort of the first 2^LOGN (threshold, unit) pairs over the threads of the block, one pair per
// thread (warp shuffles for partners within a warp, shared memory across warps; a stable total order),
// fully unrolled for the size.  Positions at or past 2^LOGN sort among themselves.
template <int LOGN>
__device__ __forceinline__ void bitonic_sort(float &key, int &idx, float *sk, int *si, int tid) {
#pragma unroll
    for (int size = 2; size <= (1 << LOGN); size <<= 1) {
#pragma unroll
        for (int stride = size >> 1; stride > 0; stride >>= 1) {
            float pk;
            int pi;
            if (stride >= 32) {
                sk[tid] = key; si[tid] = idx;
                __syncthreads();
                pk = sk[tid ^ stride]; pi = si[tid ^ stride];
                __syncthreads();
            } else {
                pk = __shfl_xor_sync(0xffffffffu, key, stride);
                pi = __shfl_xor_sync(0xffffffffu, idx, stride);
            }
            // the lower position of a pair keeps the smaller element in an ascending
            // run (the larger in a descending one); elements are distinct
            const bool keep_min = ((tid & stride) == 0) == ((tid & size) == 0);
            if (pair_less(pk, pi, key, idx) == keep_min) { key = pk; idx = pi; }
        }
    }
}

// Position of input unit `unit` (fc1 index: l*hid + k, or k when shared) in the
// per-unit arrays, which are kept in [k][l] order (k only when shared).
__device__ __forceinline__ int unit_pos(const TableLayout &lay, int unit) {
    return lay.shared ? unit : (unit % lay.hid) * lay.L + unit / lay.hid;
}

__global__ void __launch_bounds__(kPrepThreads) k_phi_prepare(luna_phi_params prm, TableLayout lay, char *table) {
    __shared__ float sk[kMaxUnits];
    __shared__ int si[kMaxUnits];
    __shared__ float w1t[kMaxUnits], b1t[kMaxUnits];  // per-unit fc1 values
    __shared__ float w2t[kMaxUnits];                  // fc2 weight of (unit k, channel l) at k*L + l
    __shared__ int tyt[kMaxUnits], rkt[kMaxUnits];
    const int tid = threadIdx.x, nt = blockDim.x;
    const int P = lay.P, N = lay.Ppad, L = lay.L, hid = lay.hid;  // N: power of two >= P, <= kMaxUnits
    float key = INFINITY;  // this thread's element: unit tid, padding (+inf, index >= P) sorts last
    int idx = tid;
    if (tid < P) {
        const float w = prm.w1[tid], c = prm.b1[tid];
        int ty;
        if (w > 0.0f) { key = up_threshold(w, c); ty = 1; }
        else if (w < 0.0f) { key = down_threshold(w, c); ty = -1; }
        else { key = INFINITY; ty = (c > 0.0f) ? -1 : 1; }  // constant unit: always on / always off
        const int tpos = unit_pos(lay, tid);
        w1t[tpos] = w; b1t[tpos] = c; tyt[tpos] = ty;
    }
    for (int e = tid; e < L * hid; e += nt) w2t[(e % hid) * L + e / hid] = prm.w2[e];  // w2[l][k]
    // bitonic sort of the first N elements (N a power of two, at most kMaxUnits = 512)
    switch (N) {
        case 2: bitonic_sort<1>(key, idx, sk, si, tid); break;
        case 4: bitonic_sort<2>(key, idx, sk, si, tid); break;
        case 8: bitonic_sort<3>(key, idx, sk, si, tid); break;
        case 16: bitonic_sort<4>(key, idx, sk, si, tid); break;
        case 32: bitonic_sort<5>(key, idx, sk, si, tid); break;
        case 64: bitonic_sort<6>(key, idx, sk, si, tid); break;
        case 128: bitonic_sort<7>(key, idx, sk, si, tid); break;
        case 256: bitonic_sort<8>(key, idx, sk, si, tid); break;
        case 512: bitonic_sort<9>(key, idx, sk, si, tid); break;
        default: break;  // N = 1: nothing to sort
    }
    sk[tid] = key;
    si[tid] = idx;
    if (idx < P) rkt[unit_pos(lay, idx)] = tid;
    __syncthreads();

    if (blockIdx.x == 0) {
        float *T = reinterpret_cast<float *>(table + lay.off_T);
        int *rank = reinterpret_cast<int *>(table + lay.off_rank);
        int *utype = reinterpret_cast<int *>(table + lay.off_utype);
        for (int r = tid; r < N; r += nt) {
            T[r] = sk[r];  // sorted kinks, +inf padding
            if (si[r] < P) rank[si[r]] = r;
        }
        for (int k = tid; k < P; k += nt) {
            const int tpos = unit_pos(lay, k);
            utype[k] = tyt[tpos];
            reinterpret_cast<float *>(table + lay.off_w1)[k] = w1t[tpos];
            reinterpret_cast<float *>(table + lay.off_b1)[k] = b1t[tpos];
        }
        for (int e = tid; e < L * hid; e += nt) reinterpret_cast<float *>(table + lay.off_w2)[e] = prm.w2[e];
        // interval search block: the sorted kinks with +inf sentinels, then every bucket's start (the
        // number of kinks strictly below the bucket's smallest value, by binary search over the kinks)
        float *Ts = reinterpret_cast<float *>(table + lay.off_Te);
        for (int e = tid; e < kSearchT; e += nt) Ts[e] = e < P ? sk[e] : INFINITY;
        unsigned short *Bk = reinterpret_cast<unsigned short *>(Ts + kSearchT);
        for (int bk = tid; bk < kBuckets; bk += nt) {
            int cnt = 0;
            if (bk > 0) {
                const int key = bucket_lo_key(bk);
                const float lo = __int_as_float(key ^ ((key >> 31) & 0x7fffffff));
                for (int step = N >> 1; step > 0; step >>= 1)  // N: power of two, +inf beyond P
                    if (sk[cnt + step - 1] < lo) cnt += step;
                if (sk[cnt] < lo) ++cnt;
            }
            Bk[bk] = (unsigned short)cnt;
        }
        for (int e = kSearchT * 2 + kBuckets + tid; e < kEytzinger * 2; e += nt)
            reinterpret_cast<unsigned short *>(Ts)[e] = 0;  // the block's unused tail
        float *W = reinterpret_cast<float *>(table + lay.off_W);
        for (int e = tid; e < lay.M * lay.d; e += nt) W[e] = prm.W[e];
        for (int e = tid; e < lay.M; e += nt) reinterpret_cast<float *>(table + lay.off_b)[e] = prm.b[e];
        for (int e = tid; e < L; e += nt) reinterpret_cast<float *>(table + lay.off_b2)[e] = prm.b2[e];
        if (lay.env) {  // envelope gate
            for (int e = tid; e < L * lay.d; e += nt) reinterpret_cast<float *>(table + lay.off_We)[e] = prm.We[e];
            for (int e = tid; e < L; e += nt) reinterpret_cast<float *>(table + lay.off_be)[e] = prm.be[e];
        }
        if (lay.coef)  // Bank+Coef coefficients
            for (int e = tid; e < L; e += nt) reinterpret_cast<float *>(table + lay.off_coef)[e] = prm.coef[e];
        if (tid == 0) {
            TableHeader *h = reinterpret_cast<TableHeader *>(table);
            h->magic = kTableMagic; h->version = kTableVersion;
            h->M = lay.M; h->L = lay.L; h->hid = lay.hid; h->d = lay.d; h->P = P; h->Ppad = lay.Ppad;
        }
    }
    // alpha, beta of (interval j, channel l), scaled by 1/sqrt(M): thread p of the
    // entry's eight sums units k = p, p + 8, ... in order, then the eight partial
    // sums are added in a fixed tree order.
    float *AB = reinterpret_cast<float *>(table + lay.off_AB);
    const float scale = 1.0f / sqrtf((float)lay.M);
    const int p = tid % kPrepSplit;
    for (int e0 = blockIdx.x * kPrepEntries; e0 < lay.nint * L; e0 += gridDim.x * kPrepEntries) {
        const int e = e0 + tid / kPrepSplit;
        const bool live = e < lay.nint * L;
        const int j = live ? e / L : 0, l = live ? e % L : 0;
        float a = 0.0f, bsum = 0.0f;
        for (int k = p; k < hid; k += kPrepSplit) {
            const int u = lay.shared ? k : k * L + l;  // the unit's kink and fc1
            const bool on = (tyt[u] > 0) ? (rkt[u] < j) : (rkt[u] >= j);
            if (on) {
                const float w2 = w2t[k * L + l];
                a = fmaf(w2, w1t[u], a);
                bsum = fmaf(w2, b1t[u], bsum);
            }
        }
#pragma unroll
        for (int o = 1; o < kPrepSplit; o <<= 1) {
            a += __shfl_xor_sync(0xffffffffu, a, o);
            bsum += __shfl_xor_sync(0xffffffffu, bsum, o);
        }
        if (live && p == 0) {
            AB[2 * e] = a * scale;
            AB[2 * e + 1] = (bsum + prm.b2[l]) * scale;
        }
    }
}

}  // namespace

cudaError_t launch_phi_prepare(const luna_phi_params &prm, const TableLayout &lay, void *table, cudaStream_t s) {
    const int blocks = (lay.nint * lay.L + kPrepEntries - 1) / kPrepEntries;
    LUNA_LAUNCH("phi_prepare", k_phi_prepare, blocks, kPrepThreads, 0, s, prm, lay, static_cast<char *>(table));
    return cudaGetLastError();
}

}  // namespace luna
