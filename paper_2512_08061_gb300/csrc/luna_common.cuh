// Internal definitions shared by the CUDA translation units of the LUNA library.
#pragma once

#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>
#include <string.h>

#include "luna.h"

namespace luna {

constexpr int kTableMagic = 0x414E554C;  // "LUNA"
constexpr int kTableVersion = 1;
constexpr int kMaxD = 128;      // max d, dv
constexpr int kMaxFeat = 128;   // max D = M * L
constexpr int kMaxL = 16;
constexpr int kMaxHidden = 128;
constexpr int kMaxUnits = 512;  // max L * hidden
constexpr int kEytzinger = 1024; // floats of the interval-search block (kept at the size of a 1023-node kink tree)

// Interval search block (4096 bytes, staged whole into shared memory by the tensor-core kernels):
//   floats [0, kSearchT)        the sorted kinks, +inf from P on (at least 16 +inf sentinels)
//   uint16 [kBuckets] after it   for each bucket of u, the number of kinks strictly below the bucket's
//                                smallest value
// A bucket is a range of an order-preserving integer key of u: 32 buckets per binade for
// 2^-7 <= |u| < 2^8, one bucket for |u| < 2^-7, and the two outer buckets extended to +-inf.  The
// interval of u (the number of kinks strictly below it) is the bucket's start plus a scan over the
// few kinks between the bucket's lower end and u; the sentinels end every scan.
constexpr int kSearchT = 528;
constexpr int kBktPos0 = 3840;                 // key >> 18 of 2^-7 (biased exponent 120, 32 per binade)
constexpr int kBktSide = 480;                  // buckets per side: 15 binades x 32
constexpr int kBktMid = kBktSide;              // the bucket of |u| < 2^-7
constexpr int kBktNeg0 = -kBktPos0 - kBktSide; // key >> 18 of the first negative bucket after the outer one
constexpr int kBuckets = 2 * kBktSide + 1;
static_assert(kSearchT * 4 + kBuckets * 2 <= kEytzinger * 4, "search block size");

// Order-preserving integer key of a float (a < b iff key(a) < key(b) for non-NaN floats other than -0/+0).
__host__ __device__ __forceinline__ int float_key(float u) {
#ifdef __CUDA_ARCH__
    const int bits = __float_as_int(u);
#else
    int bits;
    memcpy(&bits, &u, 4);
#endif
    return bits ^ ((bits >> 31) & 0x7fffffff);
}

__host__ __device__ __forceinline__ int bucket_of(float u) {
    const int kk = float_key(u) >> 18;
    if (kk >= kBktPos0) return kBktMid + 1 + (kk - kBktPos0 < kBktSide - 1 ? kk - kBktPos0 : kBktSide - 1);
    if (kk <= -kBktPos0 - 1) return kk - kBktNeg0 > 0 ? kk - kBktNeg0 : 0;
    return kBktMid;
}

// Smallest key of bucket b (b = 0: no lower end).
__host__ __device__ __forceinline__ int bucket_lo_key(int b) {
    if (b <= kBktMid - 1) return (b + kBktNeg0) * (1 << 18);
    if (b == kBktMid) return -kBktPos0 * (1 << 18);  // the first key above the negative buckets
    return (kBktPos0 + (b - kBktMid - 1)) * (1 << 18);
}

__host__ __device__ inline int next_pow2(int x) {
    int p = 1;
    while (p < x) p <<= 1;
    return p;
}
__host__ __device__ inline int64_t align16(int64_t x) { return (x + 15) & ~int64_t(15); }
__host__ __device__ inline int64_t align256(int64_t x) { return (x + 255) & ~int64_t(255); }

// Layout of the prepared feature-map table (byte offsets from its start).
//   T      [Ppad]          sorted fp32 kink thresholds of all hidden units (+inf padding)
//   Te     [1024]          the interval search block (4096 bytes): the sorted kinks with +inf sentinels
//                          and the bucket starts (see kSearchT, bucket_of)
//   AB     [nint][L][2]    per merged interval j and channel l: (alpha, beta) / sqrt(M)
//   W      [M][d], b [M]   projection copy
//   rank   [P]             position of unit (l,k) (shared MLP: unit k) in the sorted kink list
//   utype  [P]             +1: unit active iff u > T[rank] ; -1: active iff u <= T[rank]
//   w1, b1 [P], w2 [L*hid], b2 [L]  channel-MLP parameter copy (used by the gradient reduction and,
//                                    with a non-ReLU activation, by the direct evaluation)
//   We [L][d], be [L]  envelope gate (envelope variant only), coef [L] (Bank+Coef variant only)
struct TableLayout {
    int M, L, hid, d, D, P, Ppad, nint;
    int shared;  // one MLP for all channels: P = hid kinks (else P = L * hid)
    int signed_out;  // channel outputs without the outer ReLU (the listing's nonneg = False)
    int act;     // hidden-unit activation (luna_act): not ReLU = direct evaluation, no table lookup
    int env;     // envelope gate h_l(x) = sigmoid(We_l . x + be_l) on channel l
    int coef;    // Bank+Coef coefficient c_l on channel l
    int64_t off_T, off_Te, off_AB, off_W, off_b, off_rank, off_utype, off_w1, off_b1, off_w2, off_b2, bytes;
    int64_t off_We, off_be, off_coef;
};

__host__ __device__ inline TableLayout table_layout(int M, int L, int hid, int d, int shared = 0, int signed_out = 0,
                                                    int act = 0, int env = 0, int coef = 0) {
    TableLayout t;
    t.M = M; t.L = L; t.hid = hid; t.d = d; t.D = M * L;
    t.shared = shared ? 1 : 0;
    t.signed_out = signed_out ? 1 : 0;
    t.act = act;
    t.env = env ? 1 : 0;
    t.coef = coef ? 1 : 0;
    t.P = shared ? hid : L * hid;
    t.Ppad = next_pow2(t.P);
    t.nint = t.P + 1;
    int64_t o = 256;  // header
    t.off_T = o;     o = align16(o + 4 * (int64_t)t.Ppad);
    t.off_Te = o;    o = align16(o + 4 * (int64_t)kEytzinger);
    t.off_AB = o;    o = align16(o + 8 * (int64_t)t.nint * L);
    t.off_W = o;     o = align16(o + 4 * (int64_t)M * d);
    t.off_b = o;     o = align16(o + 4 * (int64_t)M);
    t.off_rank = o;  o = align16(o + 4 * (int64_t)t.P);
    t.off_utype = o; o = align16(o + 4 * (int64_t)t.P);
    t.off_w1 = o;    o = align16(o + 4 * (int64_t)t.P);
    t.off_b1 = o;    o = align16(o + 4 * (int64_t)t.P);
    t.off_w2 = o;    o = align16(o + 4 * (int64_t)L * hid);
    t.off_b2 = o;    o = align16(o + 4 * (int64_t)L);
    t.off_We = o;    o = align16(o + (t.env ? 4 * (int64_t)L * d : 0));
    t.off_be = o;    o = align16(o + (t.env ? 4 * (int64_t)L : 0));
    t.off_coef = o;  o = align16(o + (t.coef ? 4 * (int64_t)L : 0));
    t.bytes = align256(o);
    return t;
}

// Words per interval of the (alpha, beta) table in shared memory (generic kernels): 2L + 2 instead of 2L,
// so that the entries of lanes at random intervals start in 16 different 8-byte bank pairs (a 64-byte
// stride at L = 8 would put every entry in one of two) and each (alpha, beta) pair is one aligned 8-byte load.
__host__ __device__ __forceinline__ int ab_stride(const TableLayout &lay) { return 2 * lay.L + 2; }

// One of the feature-map variants (a non-ReLU activation, the envelope gate, Bank+Coef): generic kernels only.
__host__ __device__ __forceinline__ bool lay_variant(const TableLayout &lay) { return lay.act || lay.env || lay.coef; }

// Parameter-gradient partial of a block: [dW (M*d) | db (M) | MLP region | variant region].  The MLP region
// holds the interval histogram [nint][L][2] (ReLU), or with another activation the MLP gradients themselves
// [dw2 (L*hid) | dw1 (P) | db1 (P) | db2 (L)]; the variant region [dWe (L*d) | dbe (L)] (envelope) then
// [dcoef (L)] (Bank+Coef).
__host__ __device__ __forceinline__ int mlp_words(const TableLayout &lay) {
    return lay.act ? lay.L * lay.hid + 2 * lay.P + lay.L : lay.nint * lay.L * 2;
}
__host__ __device__ __forceinline__ int var_words(const TableLayout &lay) {
    return (lay.env ? lay.L * lay.d + lay.L : 0) + (lay.coef ? lay.L : 0);
}
__host__ __device__ __forceinline__ int grad_words(const TableLayout &lay) {
    return lay.M * lay.d + lay.M + mlp_words(lay) + var_words(lay);
}

struct TableHeader {
    int magic, version, M, L, hid, d, P, Ppad;
};

// ---------------------------------------------------------------------------
// I/O element access

template <typename T> struct IOType;
template <> struct IOType<float> { static constexpr luna_dtype code = LUNA_F32; };
template <> struct IOType<__nv_bfloat16> { static constexpr luna_dtype code = LUNA_BF16; };

__device__ __forceinline__ float io_load(const float *p) { return *p; }
__device__ __forceinline__ float io_load(const __nv_bfloat16 *p) { return __bfloat162float(*p); }
__device__ __forceinline__ void io_store(float *p, float v) { *p = v; }
__device__ __forceinline__ void io_store(__nv_bfloat16 *p, float v) { *p = __float2bfloat16_rn(v); }

// ---------------------------------------------------------------------------
// Feature map from the table

// Lower bound of a channel output: 0 (outer ReLU, the listing's default) or -inf (signed outputs).
// Every channel value is fmaxf(alpha u + beta, floor), and an output is active in the backward pass
// where it is above the floor.
__host__ __device__ __forceinline__ float channel_floor(const TableLayout &lay) {
    return lay.signed_out ? -INFINITY : 0.0f;
}

// Number of sorted thresholds strictly below u (branch-free lower bound over a
// power-of-two sized array whose tail is padded with +inf).
__device__ __forceinline__ int interval_of(const float *T, int Ppad, float u) {
    int pos = 0;
    for (int s = Ppad >> 1; s > 0; s >>= 1) pos += (T[pos + s - 1] < u) ? s : 0;
    pos += (T[pos] < u) ? 1 : 0;
    return pos;
}

// Interval of u from the search block (sT: its kinks, sB: its bucket starts).
__device__ __forceinline__ int interval_bucketed(const float *sT, const unsigned short *sB, float u) {
    int j = sB[bucket_of(u)];
    while (sT[j] < u) ++j;
    return j;
}

__device__ __forceinline__ int head_length(const int32_t *lengths, int b, int n) {
    if (!lengths) return n;
    int len = lengths[b];
    return len < 0 ? 0 : (len > n ? n : len);
}

// Host-side launch helpers (defined in luna_api.cu)
int device_sm_count();

}  // namespace luna
