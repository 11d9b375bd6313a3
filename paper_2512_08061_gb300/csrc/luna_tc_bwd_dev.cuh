// Device helpers shared by the tensor-core backward kernels (d = 32 and d = 64
// variants): thread layout, operand staging, the interval search and channel
// evaluation, and the fixed-point interval histogram of the channel-MLP
// gradient statistics.
#pragma once

#include "luna_tc_dev.cuh"

namespace luna {
namespace tcbwd {
namespace {  // internal linkage in every translation unit that includes this
using namespace sm100;
using namespace simt;
using namespace tcdev;

constexpr int kBWorkers = 512;           // 16 warps, four threads per row
constexpr int kBRowThreads = kBWorkers / 128;
constexpr int kBTma = 16, kBMma = 17;
constexpr int kBThreads = kBWorkers + 64;
constexpr uint32_t kBarBytes = 256;      // mbarriers, TMEM address, flag (each kernel below uses <= 26 slots)

// Projection MMA (nk 16-wide k-steps of the X tile) into TMEM.
template <class C>
__device__ __forceinline__ void proj_mma(uint32_t tmem_u, uint64_t dx, uint64_t dw) {
    constexpr uint32_t idesc = idesc_bf16(128, C::NU, false, false);
#pragma unroll
    for (int k = 0; k < C::NKD; ++k) mma_bf16_ss(tmem_u, dadd(dx, 32 * k), dadd(dw, 32 * k), idesc, k != 0);
}

// [W_hi; W_hi; W_lo; 0] as the K-major B operand of dX = [dU_hi | dU_lo | dU_hi | 0] W: row n (< d) =
// output column, K = 32 columns starting at 16-byte chunk ch0 of each 128-byte row (ch0 = 4: the upper
// half of the projection operand rows, written after stage_phi_table and a block barrier; ch0 = 0: a
// region of its own).
template <class C>
__device__ void stage_wx(const AttnArgs &a, uint8_t *dst, int ch0) {
    const float *W = reinterpret_cast<const float *>(a.table + a.lay.off_W);
    for (int e = threadIdx.x; e < C::d * 32; e += blockDim.x) {
        const int n = e / 32, k = e % 32;
        float v = 0.0f;
        if (k < 3 * C::MP) {
            __nv_bfloat16 hi, lo;
            split_bf16(W[(k % C::MP) * a.d + n], hi, lo);
            v = (k < 2 * C::MP) ? __bfloat162float(hi) : __bfloat162float(lo);
        }
        *reinterpret_cast<__nv_bfloat16 *>(dst + sw128_chunk(n, ch0 + k / 8) + (k % 8) * 2) = __float2bfloat16_rn(v);
    }
}

// Operand rows per feature (hi rows 0..D-1, lo rows D..2D-1), K = value column:
// the B operand of P = dO S^T and of dphi(k) = V dS^T.
template <class C>
__device__ void stage_rows_per_feature(const float *Sg, uint8_t *op, int tid, int nthr) {
    for (int e = tid; e < 2 * C::D * 64; e += nthr) {
        const int n = e / 64, c = e % 64, f = n % C::D;
        float v = 0.0f;
        if (c < C::DV) {
            __nv_bfloat16 hi, lo;
            split_bf16(Sg[f * C::DV + c], hi, lo);
            v = (n < C::D) ? __bfloat162float(hi) : __bfloat162float(lo);
        }
        *reinterpret_cast<__nv_bfloat16 *>(op + sw128_chunk(n, c / 8) + (c % 8) * 2) = __float2bfloat16_rn(v);
    }
}

// Operand rows per value column (hi rows 0..DV-1, lo rows DV..2DV-1), K = feature:
// the B operand of dV = phi dS.
template <class C>
__device__ void stage_rows_per_column(const float *Sg, uint8_t *op, int tid, int nthr) {
    for (int e = tid; e < 2 * C::DV * C::D; e += nthr) {
        const int n = e / C::D, f = e % C::D, c = n % C::DV;
        __nv_bfloat16 hi, lo;
        split_bf16(Sg[f * C::DV + c], hi, lo);
        *reinterpret_cast<__nv_bfloat16 *>(op + sw128_chunk(n, f / 8) + (f % 8) * 2) = (n < C::DV) ? hi : lo;
    }
}

// Interval search for the PP projections of this thread (bucketed search block).
template <int PP>
__device__ __forceinline__ void search(const float *sTe, const float (&u)[PP], int (&j)[PP]) {
    search_bucketed<PP>(sTe, u, j);
}

// alpha, beta of the 8 channels on interval j (swizzled table) and phi = max(alpha u + beta, fl): the
// outer ReLU (fl = 0) or the signed output (fl = -inf).
__device__ __forceinline__ void channel_eval(const float *sAB, int j, float u, float fl, float (&al)[8],
                                             float (&y)[8]) {
    const float4 *ab = reinterpret_cast<const float4 *>(sAB);
#pragma unroll
    for (int k = 0; k < 4; ++k) {
        const float4 v = ab[ab_slot(j, k)];
        al[2 * k] = v.x;
        al[2 * k + 1] = v.z;
        y[2 * k] = fmaxf(fmaf(v.x, u, v.y), fl);
        y[2 * k + 1] = fmaxf(fmaf(v.z, u, v.w), fl);
    }
}

// dU of two projections split into bf16 hi and lo, each pair packed into 32 bits.
__device__ __forceinline__ void dU_pack(const float (&dU)[2], uint32_t &vh, uint32_t &vl) {
    __nv_bfloat16 h0, l0, h1, l1;
    split_bf16(dU[0], h0, l0);
    split_bf16(dU[1], h1, l1);
    vh = (uint32_t)__bfloat16_as_ushort(h0) | ((uint32_t)__bfloat16_as_ushort(h1) << 16);
    vl = (uint32_t)__bfloat16_as_ushort(l0) | ((uint32_t)__bfloat16_as_ushort(l1) << 16);
}

__device__ __forceinline__ uint4 pack8(const float (&y)[8]) {
    return make_uint4(pack_bf16x2(y[0], y[1]), pack_bf16x2(y[2], y[3]), pack_bf16x2(y[4], y[5]),
                      pack_bf16x2(y[6], y[7]));
}

// Interval histogram of the channel-MLP gradient statistics: for channel l and
// interval j, the sum of g (c = 0) and of g * u (c = 1) over the samples u that
// fall into interval j, g = dLoss/dphi on an active output.
//
// Shared-memory fp32 atomics are compare-and-swap loops; int32 atomics are
// native and about five times faster.  So the bins hold fixed-point int32 sums
// over groups of hist_tiles() tiles, quantised with power-of-two scales 2^e such
// that |q| < 2^kHistQBits for the scale's reference maxima of |g| and |g*u|; a
// group holds at most 16384 samples (16 tiles of 128 rows x 8 projections,
// 8 of 128 x 16), so a bin stays below 2^30.  The
// block's first group takes its reference maxima from a pre-pass over its
// first tile with a nonzero g, every later group from the block-wide maxima of
// the group before it.  A value that does not fit (it outgrew the reference,
// or is not finite) goes, unscaled, to an fp32 atomic on the block's partial in
// global memory instead.  At the end of a group the bins are added, rescaled,
// into that partial and cleared.  The quantisation step is 2^-16 of the
// reference maximum; a sample's rounding error is at most half of it, and
// the errors of a bin's samples are independent, so a sum of N samples is off
// by about 2^-17 sqrt(N / 3) reference maxima (far below the bf16 rounding of
// the kernels' operands).  Large groups keep the block-wide flushes (a worker
// barrier and a pass over every bin) rare.
//
// Layout in shared memory: bins[(c * 8 + l) * kNint + j] (lanes with different
// intervals fall into different banks); the partial is [interval][channel][g, g*u].
__device__ __forceinline__ int hist_at(int c, int l, int j) { return (c * 8 + l) * kNint + j; }

constexpr int kHistQBits = 16;      // |q| < 2^16 per sample
constexpr int kHistSamples = 16384;  // samples per group: 16384 * 2^16 = 2^30
// Tiles per group for 128-row tiles of MP projections each.
template <int MP>
__host__ __device__ constexpr int hist_tiles() {
    static_assert(kHistSamples % (128 * MP) == 0, "whole tiles per group");
    return kHistSamples / (128 * MP);
}

// 2^e as a float, e in [-126, 127] (IEEE-754 binary32: biased exponent, zero mantissa).
__device__ __forceinline__ float pow2f(int e) { return __int_as_float((e + 127) << 23); }

// Exponent e with m * 2^e < 2^kHistQBits: m < 2^ex for ex = (biased exponent of m) - 126.
__device__ __forceinline__ int hist_exp_of(float m) {
    const int ex = (int)((__float_as_uint(m) >> 23) & 255u) - 126;
    return max(-126, min(126, kHistQBits - ex));
}

// Block-uniform state of the fixed-point bins.
struct HistAcc {
    int e0 = 0, e1 = 0;        // exponents of the current group
    int tiles = 0;             // tiles of the current group added so far
    bool open = false;         // scales known (from the first nonzero tile, then from the previous group)
    float m0 = 0.f, m1 = 0.f;  // this thread's maxima of the finite |g|, |g*u| added to the current group
};

// Running maximum of the finite |v|.
__device__ __forceinline__ float finite_max(float m, float v) {
    const float a = fabsf(v);
    return a <= 3.402823466e38f ? fmaxf(m, a) : m;
}

// Block-wide maxima of the workers' m0, m1 (one worker barrier; smax holds
// 2 * (kBWorkers / 32) floats and is written again only after a later worker
// barrier), then the scales: false (scales unchanged) when both are zero.
__device__ __forceinline__ bool hist_scales(HistAcc &h, float m0, float m1, float *smax, int warp, int lane) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        m0 = fmaxf(m0, __shfl_xor_sync(0xffffffffu, m0, o));
        m1 = fmaxf(m1, __shfl_xor_sync(0xffffffffu, m1, o));
    }
    constexpr int NW = kBWorkers / 32;
    if (lane == 0) { smax[warp] = m0; smax[NW + warp] = m1; }
    named_sync<kBWorkers>(1);
    m0 = 0.0f;
    m1 = 0.0f;
#pragma unroll
    for (int w = 0; w < NW; ++w) { m0 = fmaxf(m0, smax[w]); m1 = fmaxf(m1, smax[NW + w]); }
    if (m0 == 0.0f && m1 == 0.0f) return false;
    h.e0 = hist_exp_of(m0 > 0.0f ? m0 : m1);
    h.e1 = hist_exp_of(m1 > 0.0f ? m1 : m0);
    return true;
}

// Opens the first group of the block from this thread's maxima over its first
// tile (a pre-pass); later groups take their scales from the previous group.
// Returns false while every g seen so far is zero.
__device__ __forceinline__ bool hist_open(HistAcc &h, float m0, float m1, float *smax, int warp, int lane) {
    h.open = hist_scales(h, m0, m1, smax, warp, lane);
    return h.open;
}

// Adds value v of (c, l) for a sample in interval j: int32 bin if it fits the
// group's scale s, else an fp32 atomic on the global partial.
__device__ __forceinline__ void hist_put(int *bins, float *part, int c, int l, int j, float v, float s) {
    if (v != 0.0f) {
        const float q = v * s;
        if (fabsf(q) < (float)(1 << kHistQBits))
            atomicAdd(bins + hist_at(c, l, j), __float2int_rn(q));
        else
            atomicAdd(part + ((j * 8 + l) << 1) + c, v);
    }
}

// The per-value path of hist_add for a sample some of whose values outgrew the
// group's scales (or are not finite): rare, so it stays out of line and the
// common path keeps the kernels' loops small in the instruction cache.  The
// values come by value (an array argument would move the caller's array to
// local memory).
__device__ __noinline__ void hist_add_slow(int *bins, float *part, int j, float u, float s0, float s1, float g0,
                                           float g1, float g2, float g3, float g4, float g5, float g6, float g7) {
    const float g[8] = {g0, g1, g2, g3, g4, g5, g6, g7};
#pragma unroll
    for (int l = 0; l < 8; ++l) {
        hist_put(bins, part, 0, l, j, g[l], s0);
        hist_put(bins, part, 1, l, j, g[l] * u, s1);
    }
}

// x * s rounded to the nearest integer (ties to even), for |x s| < 2^22: one
// fused multiply-add onto 1.5 * 2^23, where the float spacing is 1, rounds the
// exact product once; the integer is then the low bits of the sum.  Same
// result as __float2int_rn(x * s) for a power-of-two s, without the
// conversion unit.
__device__ __forceinline__ int round_scaled(float x, float s) {
    return __float_as_int(fmaf(x, s, 12582912.0f)) - 0x4B400000;
}

// Adds the tile's samples (8 channel values g each, zero where inactive, and
// du = sum_l g_l alpha_l) to the bins and tracks this thread's maxima for the
// next group's scales.  A sample whose largest |g| and |g u| fit the group's
// scales and whose du is finite (so no g is NaN or infinite) takes the fast
// path: every value fits, so the per-value range test is skipped.  The scales
// are powers of two, so g * (u s1) equals (g u) s1 exactly.
template <int PP>
__device__ __forceinline__ void hist_add(int *bins, float *part, HistAcc &h, const int (&j)[PP],
                                         const float (&u)[PP], const float (&g)[PP][8], const float (&du)[PP]) {
    const float s0 = pow2f(h.e0), s1 = pow2f(h.e1);
    constexpr float kQ = (float)(1 << kHistQBits);
#pragma unroll
    for (int q = 0; q < PP; ++q) {
        float mg = 0.0f;
#pragma unroll
        for (int l = 0; l < 8; ++l) mg = fmaxf(mg, fabsf(g[q][l]));
        const float mgu = mg * fabsf(u[q]);
        h.m0 = finite_max(h.m0, mg);
        h.m1 = finite_max(h.m1, mgu);
        if (mg * s0 < kQ && mgu * s1 < kQ && du[q] - du[q] == 0.0f) {
            const float us1 = u[q] * s1;
#pragma unroll
            for (int l = 0; l < 8; ++l)
                if (g[q][l] != 0.0f) {
                    atomicAdd(bins + hist_at(0, l, j[q]), round_scaled(g[q][l], s0));
                    atomicAdd(bins + hist_at(1, l, j[q]), round_scaled(g[q][l], us1));
                }
        } else {
            hist_add_slow(bins, part, j[q], u[q], s0, s1, g[q][0], g[q][1], g[q][2], g[q][3], g[q][4], g[q][5],
                          g[q][6], g[q][7]);
        }
    }
}

// Closes the group: after a worker barrier (every atomic done), adds the bins,
// rescaled, into the partial and clears them (thread t handles entries t,
// t + kBWorkers, ...); with `next`, the group's block-wide maxima then give the
// scales of the next group (unchanged if it was all zero).
__device__ __forceinline__ void hist_close(int *bins, float *part, int nint, HistAcc &h, int t, bool next,
                                           float *smax, int warp, int lane) {
    named_sync<kBWorkers>(1);
    const float inv0 = pow2f(-h.e0), inv1 = pow2f(-h.e1);
#pragma unroll 4
    for (int e = t; e < nint * 16; e += kBWorkers) {
        const int at = hist_at(e & 1, (e >> 1) & 7, e >> 4);
        const int v = bins[at];
        bins[at] = 0;
        part[e] = __ldcg(part + e) + (float)v * ((e & 1) ? inv1 : inv0);  // L2 copy: fp32 atomics went there
    }
    if (next) hist_scales(h, h.m0, h.m1, smax, warp, lane);
    h.tiles = 0;
    h.m0 = h.m1 = 0.0f;
}

// Zeroes a row of a 128-row x 128 B tile (padded rows must not carry garbage
// into contractions over rows).
__device__ __forceinline__ void zero_row(uint8_t *tile, int r) {
#pragma unroll
    for (int c = 0; c < 8; ++c) *reinterpret_cast<uint4 *>(tile + sw128_chunk(r, c)) = make_uint4(0, 0, 0, 0);
}

// Writes dW (M x d, from smem) and db (block sum of per-thread values) into the
// block's parameter-gradient partial; its histogram part is written tile by tile.
template <class C>
__device__ void store_param_partial(const AttnArgs &a, const float *sdW, float *sdb, float *gp) {
    const int Md = C::MP * a.d;
    for (int e = threadIdx.x; e < Md; e += blockDim.x) gp[e] = sdW[e];
    for (int e = threadIdx.x; e < C::MP; e += blockDim.x) gp[Md + e] = sdb[e];
}

}  // namespace
}  // namespace tcbwd
}  // namespace luna
