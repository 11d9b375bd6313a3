// Device helpers shared by the tensor-core kernels (forward and backward).
#pragma once

#include <math.h>
#include <stdlib.h>

#include "luna_prof.cuh"
#include "luna_sm100.cuh"
#include "luna_simt_dev.cuh"
#include "luna_tc.cuh"

namespace luna {
namespace tcdev {
namespace {  // internal linkage in every translation unit that includes this
using namespace sm100;
using namespace simt;

constexpr uint32_t kSmemLimit = 227 * 1024;
constexpr int kPpad = 512;   // merged kink list (L * hidden <= 512, L = 8)
constexpr int kNint = 513;   // intervals
constexpr uint32_t kTableBytes = (kEytzinger + kNint * 16 + 32) * 4;

// Intervals of the PP values u (the number of kinks strictly below each) from the interval search block
// in shared memory (sS: its sorted kinks, then its bucket starts): the bucket starts of all PP values,
// one scan step for all of them (most buckets hold at most one kink below u), then the rest of each scan,
// rarely more than one step more.  Exact for every non-NaN u (the sentinels end each scan).
template <int PP>
__device__ __forceinline__ void search_bucketed(const float *sS, const float (&u)[PP], int (&j)[PP]) {
    const unsigned short *sB = reinterpret_cast<const unsigned short *>(sS + kSearchT);
#pragma unroll
    for (int q = 0; q < PP; ++q) j[q] = sB[bucket_of(u[q])];
#pragma unroll
    for (int q = 0; q < PP; ++q) j[q] += sS[j[q]] < u[q] ? 1 : 0;
#pragma unroll
    for (int q = 0; q < PP; ++q)
        while (sS[j[q]] < u[q]) ++j[q];
}

// First 1024-byte boundary at or after p (a shared-memory array), formed by
// pointer arithmetic on p so that the compiler still sees a shared address.
__device__ __forceinline__ uint8_t *align1024(uint8_t *p) {
    return p + ((1024u - (smem_u32(p) & 1023u)) & 1023u);
}

__device__ __forceinline__ uint32_t pack_bf16x2(float a, float b) {
    __nv_bfloat162 v = __floats2bfloat162_rn(a, b);
    return *reinterpret_cast<uint32_t *>(&v);
}

__device__ __forceinline__ void split_bf16(float x, __nv_bfloat16 &hi, __nv_bfloat16 &lo) {
    hi = __float2bfloat16_rn(x);
    lo = __float2bfloat16_rn(x - __bfloat162float(hi));
}

__device__ __forceinline__ void report(int *status, int code) {
    if (status) atomicOr(status, code);
}

// Bounded wait that turns into a no-op once this thread has seen a timeout, so
// that every thread still runs the same sequence of block-level barriers and
// the kernel terminates (its outputs are then undefined and the status word
// reports LUNA_ERR_DEVICE_TIMEOUT).
__device__ __forceinline__ void wait_or_fail(uint64_t *bar, uint32_t parity, bool &failed, int *status) {
    if (failed) return;
    if (!mbar_wait(bar, parity)) {
        failed = true;
        report(status, 1);
    }
}

template <int N>
__device__ __forceinline__ void named_sync(int id) {
    asm volatile("bar.sync %0, %1;" ::"r"(id), "r"(N) : "memory");
}

// Barrier of the four worker warps w, w + 4, w + 8, w + 12 that share TMEM lane quarter w % 4 (the threads
// of the same rows): named barriers 3..6, so that the quarters of a tile run independently.
__device__ __forceinline__ void quarter_sync(int warp) {
    asm volatile("bar.sync %0, 128;" ::"r"(3 + (warp & 3)) : "memory");
}

// Adds a byte offset to the start-address field of a shared-memory descriptor.
__device__ __forceinline__ uint64_t dadd(uint64_t desc, uint32_t bytes) { return desc + (bytes >> 4); }

// Slot of float4 k (channels 2k, 2k+1: alpha, beta, alpha, beta) of interval j
// in the shared interval table.  Lanes read rows j at random; the XOR with bits
// 1-2 of j spreads the 16-byte reads of a warp over all eight 16-byte bank
// groups (bit 0 of j already selects the upper or lower half of a 128-byte line).
__device__ __forceinline__ int ab_slot(int j, int k) { return (j << 2) | (k ^ ((j >> 1) & 3)); }

// Loads the breadth-first kink list, the interval table (slots ab_slot) and the
// projection bias into smem, and writes the
// projection operand (NU rows x DX, K-major SW128): W split into bf16 terms
// W_hi + W_mid (NU = 2M, about 16 significant bits) or W_hi + W_mid + W_lo and
// M zero rows (NU = 4M, about 24 bits, as fp32).
template <class C>
__device__ void stage_phi_table(const AttnArgs &a, float *sTe, float *sAB, float *sbias, uint8_t *Wop) {
    const int tid = threadIdx.x, nthreads = blockDim.x;
    const TableLayout &lay = a.lay;
    const float4 *Te4 = reinterpret_cast<const float4 *>(a.table + lay.off_Te);
    for (int e = tid; e < kEytzinger / 4; e += nthreads) reinterpret_cast<float4 *>(sTe)[e] = Te4[e];
    const float4 *AB4 = reinterpret_cast<const float4 *>(a.table + lay.off_AB);
#pragma unroll 4
    for (int e = tid; e < lay.nint * 4; e += nthreads) {
        const int j = e >> 2, k = e & 3;
        reinterpret_cast<float4 *>(sAB)[ab_slot(j, k)] = AB4[e];
    }
    const float *b = reinterpret_cast<const float *>(a.table + lay.off_b);
    for (int e = tid; e < C::MP; e += nthreads) sbias[e] = b[e];
    const float *W = reinterpret_cast<const float *>(a.table + lay.off_W);
    for (int e = tid; e < C::NU * C::DX; e += nthreads) {
        const int n = e / C::DX, c = e % C::DX;
        const int i = n % C::MP, part = n / C::MP;  // rows: W_hi, W_mid[, W_lo, 0]
        const float w = (c < a.d) ? W[i * a.d + c] : 0.0f;
        const __nv_bfloat16 hi = __float2bfloat16_rn(w);
        const float r1 = w - __bfloat162float(hi);
        const __nv_bfloat16 mid = __float2bfloat16_rn(r1);
        const __nv_bfloat16 lo = __float2bfloat16_rn(r1 - __bfloat162float(mid));
        *reinterpret_cast<__nv_bfloat16 *>(Wop + (c / 64) * (C::NU * 128) + sw128_chunk(n, (c % 64) / 8) + (c % 8) * 2) =
            part == 0 ? hi : part == 1 ? mid : part == 2 ? lo : __float2bfloat16_rn(0.0f);
    }
}

// Work decomposition shared by the persistent kernels: item = (head, chunk of
// a.rows_per_split rows); block c walks the contiguous item range
// [c*items/G, (c+1)*items/G), so consecutive items mostly share a head.
struct Items {
    int nchunk, rows, total, begin, end;
    __device__ Items(const AttnArgs &a) {
        rows = a.rows_per_split;
        nchunk = a.nsplit;
        total = a.B * a.H * nchunk;
        if (a.split) {  // balanced by valid tiles (padded sequences)
            begin = a.split[blockIdx.x];
            end = a.split[blockIdx.x + 1];
        } else {
            begin = (int)((long long)blockIdx.x * total / gridDim.x);
            end = (int)((long long)(blockIdx.x + 1) * total / gridDim.x);
        }
    }
};

struct ItemRange {
    int bh, chunk, r0, rend, r1, ntiles;
};

__device__ __forceinline__ ItemRange item_range(const AttnArgs &a, const Items &it, int item) {
    ItemRange g;
    g.bh = item / it.nchunk;
    g.chunk = item - g.bh * it.nchunk;
    const int len = head_length(a.lengths, g.bh / a.H, a.n);
    g.r0 = g.chunk * it.rows;
    g.rend = min(a.n, g.r0 + it.rows);
    g.r1 = min(len, g.rend);
    g.ntiles = g.r1 > g.r0 ? (g.r1 - g.r0 + 127) / 128 : 0;
    return g;
}

// The blocks that own items of head bh (a contiguous block range): how many
// there are, and how many of them come before this block.
struct RunSlot {
    int rank, nruns;
};

__device__ __forceinline__ RunSlot run_slot(const AttnArgs &a, const Items &it, int bh) {
    if (a.runs) return RunSlot{(int)blockIdx.x - a.runs[2 * bh], a.runs[2 * bh + 1] - a.runs[2 * bh] + 1};
    const long long total = it.total;
    const int G = gridDim.x;
    const int c_first = (int)((((long long)bh * it.nchunk + 1) * G - 1) / total);
    const int c_last = (int)((((long long)(bh + 1) * it.nchunk) * G - 1) / total);
    return RunSlot{(int)blockIdx.x - c_first, c_last - c_first + 1};
}

// out[e] = sum_{p < np} part[p][e] in order p = 0..np-1, for e < count
// (count % 4 == 0), by `nthr` threads (this one is number t): float4 loads of
// up to four partials are in flight before they are added.
__device__ __forceinline__ void ordered_sum4(const float *part, int np, int count, float *out, int t, int nthr) {
    for (int e = 4 * t; e < count; e += 4 * nthr) {
        float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
        for (int p0 = 0; p0 < np; p0 += 4) {
            float4 v[4];
#pragma unroll
            for (int k = 0; k < 4; ++k)
                if (p0 + k < np) v[k] = __ldcg(reinterpret_cast<const float4 *>(part + (size_t)(p0 + k) * count + e));
#pragma unroll
            for (int k = 0; k < 4; ++k)
                if (p0 + k < np) { acc.x += v[k].x; acc.y += v[k].y; acc.z += v[k].z; acc.w += v[k].w; }
        }
        *reinterpret_cast<float4 *>(out + e) = acc;
    }
}

// Iterates the flattened (item, tile) sequence of a block.
struct TileCursor {
    int item, t;
    ItemRange g;
    __device__ void start(const AttnArgs &a, const Items &it) {
        item = it.begin;
        t = 0;
        if (item < it.end) g = item_range(a, it, item);
        skip(a, it);
    }
    __device__ void skip(const AttnArgs &a, const Items &it) {
        while (item < it.end && t >= g.ntiles) {
            ++item;
            t = 0;
            if (item < it.end) g = item_range(a, it, item);
        }
    }
    __device__ void next(const AttnArgs &a, const Items &it) {
        ++t;
        skip(a, it);
    }
    __device__ int row0() const { return g.r0 + t * 128; }
};

__device__ __forceinline__ int block_tiles(const AttnArgs &a, const Items &it) {
    int T = 0;
    for (int i = it.begin; i < it.end; ++i) T += item_range(a, it, i).ntiles;
    return T;
}


}  // namespace
}  // namespace tcdev
}  // namespace luna
