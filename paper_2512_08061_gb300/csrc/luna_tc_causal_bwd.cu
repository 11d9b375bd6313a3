// Backward pass of the streaming (causal) form on tensor cores (bf16 I/O,
// d = dv = 128, M = 16 projections, L = 8 channels: D = 128 features).
//
// With S_i = sum_{j<=i} phi(k_j) v_j^T, z_i = sum_{j<=i} phi(k_j),
// den_i = phi(q_i).z_i + eps and O_i = phi(q_i)^T S_i / den_i (Eq. kernel-attn
// in its streaming form), the gradient given dO is
//   P_i = S_i dO_i,  ndot_i = -(dO_i . O_i) = -phi(q_i).P_i / den_i
//   dphi(q_i) = (P_i + z_i ndot_i) / den_i
//   dS_j = sum_{i>=j} phi~(q_i) dO_i^T,  dz_j = sum_{i>=j} phi~(q_i) ndot_i,  phi~ = phi / den
//   dv_j = dS_j^T phi(k_j),  dphi(k_j) = dS_j v_j + dz_j
// followed by the chain rule through the feature map (luna_tc_phi_bwd.cu).
//
// The rows of a head are cut into the state segments of the forward pass;
// inside a segment the kernels walk 64-row tiles with the running state in
// tensor memory.  Stages:
//   1. k_tcc_query (forward sweep, state S, z from the segment prefixes):
//        MMA  U = [Q | K] [W_hi; W_mid]^T        -> phi(q) (fp32), phi(k) (bf16 hi + lo tiles)
//        MMA  F = dO V^T,  Zc = L phi(K) (L lower-triangular ones),  P = dO [S_hi; S_lo]^T
//        work z_i = z + Zc_i, den_i, F masked to j <= i (hi + lo)
//        MMA  P += F_masked phi(K),  S += phi(K)^T V,  z += phi(K)^T 1
//        work ndot_i, dphi(q_i); writes dphi(q), phi(k) (hi, lo), phi~(q) (hi, lo), (den, ndot)
//   2. k_tcc_dstats: per segment sum_i phi~(q_i) dO_i^T and sum_i phi~(q_i) ndot_i
//   3. k_seg_rscan: exclusive suffix of those sums (dS, dz after each segment)
//   4. k_tcc_key (reverse sweep, state dS, dz in tensor memory):
//        MMA  C = phi(K) phi~(Q)^T,  E = V dO^T
//        work C masked to i >= j (hi + lo); E + ndot_i masked (hi + lo)
//        MMA  dV = phi(K) [dS_hi; dS_lo] + C dO,  dphi = V [dS_hi; dS_lo]^T + E phi~(Q)
//             dS += phi~(Q)^T dO,  dz += phi~(Q)^T [ndot_hi, ndot_lo]
//        work dV, dphi(k) = dphi + dz
//   5. chain rule for Q and for K, then the parameter-gradient reduction.
// Precision: dO and V enter exactly; everything else as a bf16 hi + lo pair (the
// states, phi(k), phi~(q), the masked score tiles; a product of two pairs drops
// lo x lo).  When the features vary little between tokens, P_i and z_i (dO_i .
// O_i) cancel to a few percent of either, so a single bf16 rounding of phi(k)
// in the tile-local terms would cost tens of percent of dphi(q); ndot is taken
// from the same P as dphi(q), so that this cancellation is exact up to rounding.
#include "luna_tc_dev.cuh"

namespace luna {
namespace {
using namespace sm100;
using namespace simt;
using namespace tcdev;

constexpr int kCBWorkers = 512;  // 16 warps: warp w covers rows 16*(w%4) .. +15 and column group w/4
constexpr int kCBTma = 16, kCBMma = 17;
constexpr int kCBThreads = kCBWorkers + 64;

struct K64 {
    static constexpr int d = 128, DX = 128, DV = 128, MP = 16, D = 128, NU = 32;
    static constexpr uint32_t T8 = 8192;    // 64 rows x 128 B (one 64-column block of a 64-row tile)
    static constexpr uint32_t T16 = 16384;  // 128 rows x 128 B
    static constexpr uint32_t RT = 2 * T8;  // a 64-row tile of 128 columns
    static constexpr uint32_t SOP = 2 * T16;  // state operand [feature][value], 128 x 128
    static constexpr uint32_t WOP = 2 * NU * 128;
    // query side
    static constexpr uint32_t SMEM_Q = 5 * RT + 3 * T8 + 2 * SOP + 2048 + WOP + kTableBytes + 2 * D * 4 +
                                       2 * 8 * 64 * 4 + 256 + 1024;
    // key side
    static constexpr uint32_t SMEM_K = 2 * RT + 2 * RT + RT + RT + 2048 + 4 * T8 + 2 * SOP + D * 4 + 256 + 1024;
    static_assert(SMEM_Q <= kSmemLimit && SMEM_K <= kSmemLimit, "shared memory budget");
};

// 64-row tiles of the work items (state segments) of a block.
__device__ __forceinline__ int tiles64(const ItemRange &g) { return g.r1 > g.r0 ? (g.r1 - g.r0 + 63) / 64 : 0; }

__device__ __forceinline__ int block_tiles64(const AttnArgs &a, const Items &it) {
    int T = 0;
    for (int i = it.begin; i < it.end; ++i) T += tiles64(item_range(a, it, i));
    return T;
}

// Walks the (item, tile) sequence of a block; within an item the tiles run
// forward (rev = false) or backward.
struct Cursor64 {
    int item, t, nt;
    ItemRange g;
    bool rev;
    __device__ void start(const AttnArgs &a, const Items &it, bool reverse) {
        rev = reverse;
        item = it.begin;
        t = 0;
        nt = 0;
        if (item < it.end) { g = item_range(a, it, item); nt = tiles64(g); }
        skip(a, it);
    }
    __device__ void skip(const AttnArgs &a, const Items &it) {
        while (item < it.end && t >= nt) {
            ++item;
            t = 0;
            if (item < it.end) { g = item_range(a, it, item); nt = tiles64(g); }
        }
    }
    __device__ void next(const AttnArgs &a, const Items &it) { ++t; skip(a, it); }
    __device__ int tile() const { return rev ? nt - 1 - t : t; }
    __device__ int row0() const { return g.r0 + 64 * tile(); }
};

// M = 64 accumulators: row m lives in lane 32*(m/16) + m%16.  A warp loads 2N
// columns of its 16 rows (threads 0-15 hold them); thread t < 16 keeps the first
// N, thread t + 16 receives the last N of thread t.
template <int N>
__device__ __forceinline__ void half_cols(const uint32_t (&x)[2 * N], float (&mine)[N], int lane) {
#pragma unroll
    for (int k = 0; k < N; ++k) {
        const uint32_t b = __shfl_sync(0xffffffffu, x[N + k], lane & 15);
        mine[k] = __uint_as_float(lane < 16 ? x[k] : b);
    }
}

__device__ __forceinline__ void ld32(uint32_t taddr, uint32_t (&x)[32]) {
    uint32_t a[16], b[16];
    tmem_ld16(taddr, a);
    tmem_ld16(taddr + 16, b);
    tmem_wait_ld();
#pragma unroll
    for (int k = 0; k < 16; ++k) { x[k] = a[k]; x[16 + k] = b[k]; }
}

// 32 fp32 values -> bf16 hi and lo rows of a state operand [feature][value]
// (value blocks of 64 columns T16 bytes apart), feature row f, columns c0 .. c0+31.
__device__ __forceinline__ void store_state32(uint8_t *hi, uint8_t *lo, int f, int c0, const float (&v)[32]) {
    const uint32_t blk = (uint32_t)(c0 / 64) * K64::T16;
    const int ch0 = (c0 % 64) / 8;
#pragma unroll
    for (int k = 0; k < 4; ++k) {
        uint32_t wh[4], wl[4];
#pragma unroll
        for (int e = 0; e < 4; ++e) {
            __nv_bfloat16 h0, l0, h1, l1;
            split_bf16(v[8 * k + 2 * e], h0, l0);
            split_bf16(v[8 * k + 2 * e + 1], h1, l1);
            wh[e] = (uint32_t)__bfloat16_as_ushort(h0) | ((uint32_t)__bfloat16_as_ushort(h1) << 16);
            wl[e] = (uint32_t)__bfloat16_as_ushort(l0) | ((uint32_t)__bfloat16_as_ushort(l1) << 16);
        }
        *reinterpret_cast<uint4 *>(hi + blk + sw128_chunk(f, ch0 + k)) = make_uint4(wh[0], wh[1], wh[2], wh[3]);
        *reinterpret_cast<uint4 *>(lo + blk + sw128_chunk(f, ch0 + k)) = make_uint4(wl[0], wl[1], wl[2], wl[3]);
    }
}

// Eight values -> bf16 hi and lo chunks.
__device__ __forceinline__ void split8(const float (&v)[8], uint4 &h, uint4 &l) {
    uint32_t wh[4], wl[4];
#pragma unroll
    for (int e = 0; e < 4; ++e) {
        __nv_bfloat16 h0, l0, h1, l1;
        split_bf16(v[2 * e], h0, l0);
        split_bf16(v[2 * e + 1], h1, l1);
        wh[e] = (uint32_t)__bfloat16_as_ushort(h0) | ((uint32_t)__bfloat16_as_ushort(h1) << 16);
        wl[e] = (uint32_t)__bfloat16_as_ushort(l0) | ((uint32_t)__bfloat16_as_ushort(l1) << 16);
    }
    h = make_uint4(wh[0], wh[1], wh[2], wh[3]);
    l = make_uint4(wl[0], wl[1], wl[2], wl[3]);
}

__device__ __forceinline__ uint4 pack8f(const float *y) {
    return make_uint4(pack_bf16x2(y[0], y[1]), pack_bf16x2(y[2], y[3]), pack_bf16x2(y[4], y[5]),
                      pack_bf16x2(y[6], y[7]));
}

// ---------------------------------------------------------------------------
// 1. query side

template <class C, bool TSUM>  // TSUM: also sum phi . dphi per channel into tpart (channel normalisation)
__global__ void __launch_bounds__(kCBThreads, 1)
    k_tcc_query(const __grid_constant__ CUtensorMap mapQ, const __grid_constant__ CUtensorMap mapK,
                const __grid_constant__ CUtensorMap mapV, const __grid_constant__ CUtensorMap mapdO, AttnArgs a,
                double *tpart, int *status) {
    extern __shared__ uint8_t smem_raw[];
    uint8_t *sm = align1024(smem_raw);
    constexpr uint32_t T8 = C::T8, RT = C::RT;
    uint8_t *Qb = sm;
    uint8_t *Kb = Qb + RT;           // K, then (once projected) phi(K) hi, [key][feature]
    uint8_t *Vb = Kb + RT;
    uint8_t *Ob = Vb + RT;           // dO
    uint8_t *Pk = Ob + RT;           // phi(K) lo
    uint8_t *Fh = Pk + RT;           // masked F, hi and lo ([query][key])
    uint8_t *Fl = Fh + T8;
    uint8_t *L1 = Fl + T8;           // lower-triangular ones [query][key]
    uint8_t *Sh = L1 + T8;           // state operand [feature][value], hi and lo
    uint8_t *Sl = Sh + C::SOP;
    uint8_t *Ones = Sl + C::SOP;     // 16 rows x 64 keys
    uint8_t *Wop = Ones + 2048;
    float *sTe = reinterpret_cast<float *>(Wop + C::WOP);
    float *sAB = sTe + kEytzinger;
    float *sbias = sAB + kNint * 16;
    float *sz = sbias + 32;          // z before the current tile
    float *zpre = sz + C::D;         // z at the segment start
    float *sred = zpre + C::D;       // [den, dot][8 parts][64 rows]
    uint64_t *bars = reinterpret_cast<uint64_t *>(sred + 2 * 8 * 64);
    uint64_t *fullx = bars, *fullvo = bars + 2, *infree = bars + 3;
    uint64_t *uready = bars + 4, *phiready = bars + 5, *sopready = bars + 6, *aready = bars + 7;
    uint64_t *fready = bars + 8, *pready = bars + 9, *sready = bars + 10;
    uint32_t *tslot = reinterpret_cast<uint32_t *>(bars + 11);

    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const Items it(a);
    // TMEM: U (then F) [64] | Zc [128] | P [128] | S [128] | z [16]
    constexpr uint32_t cU = 0, cZc = 64, cP = 192, cS = 320, cz = 448;

    if (tid == 0) {
        mbar_init(fullx, 1); mbar_init(fullvo, 1); mbar_init(infree, 1);
        mbar_init(uready, 1); mbar_init(phiready, kCBWorkers); mbar_init(sopready, kCBWorkers);
        mbar_init(aready, 1); mbar_init(fready, kCBWorkers); mbar_init(pready, 1); mbar_init(sready, 1);
        fence_mbar_init();
    }
    if (warp == 0) { tmem_alloc(tslot, 512); tmem_relinquish(); }
    stage_phi_table<C>(a, sTe, sAB, sbias, Wop);
    for (int e = tid; e < 64 * 8; e += blockDim.x) {  // L: row i has ones at keys j <= i
        const int i = e / 8, c = e % 8;
        uint32_t w[4];
#pragma unroll
        for (int k = 0; k < 4; ++k) {
            const int j0 = 8 * c + 2 * k;
            w[k] = (j0 <= i ? 0x3F80u : 0u) | ((j0 + 1 <= i ? 0x3F80u : 0u) << 16);
        }
        *reinterpret_cast<uint4 *>(L1 + sw128_chunk(i, c)) = make_uint4(w[0], w[1], w[2], w[3]);
    }
    for (int e = tid; e < 2048 / 4; e += blockDim.x) reinterpret_cast<uint32_t *>(Ones)[e] = 0x3F803F80u;
    // rows of the items beyond the sequence length: zero phi(k), phi~(q) (read by later stages)
    for (int item = it.begin; item < it.end; ++item) {
        const ItemRange ir = item_range(a, it, item);
        const int z0 = max(ir.r0, ir.r1);
        uint4 *pk = reinterpret_cast<uint4 *>(static_cast<__nv_bfloat16 *>(a.phik) + ((size_t)ir.bh * a.n + z0) * 2 * C::D);
        uint4 *pq = reinterpret_cast<uint4 *>(static_cast<__nv_bfloat16 *>(a.pq2) + ((size_t)ir.bh * a.n + z0) * 2 * C::D);
        for (int e = tid; e < (ir.rend - z0) * 2 * C::D / 8; e += blockDim.x) pk[e] = make_uint4(0, 0, 0, 0);
        for (int e = tid; e < (ir.rend - z0) * 2 * C::D / 8; e += blockDim.x) pq[e] = make_uint4(0, 0, 0, 0);
    }
    fence_proxy_async_smem();
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tbase = *tslot;
    const int T = block_tiles64(a, it);

    if (warp == kCBTma) {
        if (lane < 2) {
            Cursor64 cur;
            cur.start(a, it, false);
            bool failed = false;
            for (int g = 0; g < T && !failed; ++g, cur.next(a, it)) {
                if (lane == 0) {  // the K buffer holds phi(K) hi until the tile's last contraction
                    if (g >= 1) wait_or_fail(infree, (g - 1) & 1, failed, status);
                    mbar_arrive_expect_tx(fullx, 2 * RT);
                    for (int kb = 0; kb < 2; ++kb) {
                        tma_load_3d(Qb + kb * T8, &mapQ, kb * 64, cur.row0(), cur.g.bh, fullx);
                        tma_load_3d(Kb + kb * T8, &mapK, kb * 64, cur.row0(), cur.g.bh, fullx);
                    }
                } else {
                    if (g >= 1) wait_or_fail(infree, (g - 1) & 1, failed, status);
                    mbar_arrive_expect_tx(fullvo, 2 * RT);
                    for (int kb = 0; kb < 2; ++kb) {
                        tma_load_3d(Vb + kb * T8, &mapV, kb * 64, cur.row0(), cur.g.bh, fullvo);
                        tma_load_3d(Ob + kb * T8, &mapdO, kb * 64, cur.row0(), cur.g.bh, fullvo);
                    }
                }
            }
        }
    } else if (warp == kCBMma) {
        if (lane == 0) {
            const uint64_t dQk = sdesc(smem_u32(Qb), 16, 1024, kSwizzle128);
            const uint64_t dKk = sdesc(smem_u32(Kb), 16, 1024, kSwizzle128);
            const uint64_t dVk = sdesc(smem_u32(Vb), 16, 1024, kSwizzle128);     // K-major, rows = keys
            const uint64_t dVm = sdesc(smem_u32(Vb), T8, 1024, kSwizzle128);     // MN-major, N = values
            const uint64_t dOk = sdesc(smem_u32(Ob), 16, 1024, kSwizzle128);     // K-major, rows = queries
            const uint64_t dKm = sdesc(smem_u32(Kb), T8, 1024, kSwizzle128);     // phi(K) hi, MN-major, M/N = features
            const uint64_t dPm = sdesc(smem_u32(Pk), T8, 1024, kSwizzle128);     // phi(K) lo
            const uint64_t dFh = sdesc(smem_u32(Fh), 16, 1024, kSwizzle128);
            const uint64_t dFl = sdesc(smem_u32(Fl), 16, 1024, kSwizzle128);
            const uint64_t dL1 = sdesc(smem_u32(L1), 16, 1024, kSwizzle128);
            const uint64_t dSh = sdesc(smem_u32(Sh), 16, 1024, kSwizzle128);     // K-major, rows = features
            const uint64_t dSl = sdesc(smem_u32(Sl), 16, 1024, kSwizzle128);
            const uint64_t dW = sdesc(smem_u32(Wop), 16, 1024, kSwizzle128);
            const uint64_t d1 = sdesc(smem_u32(Ones), 16, 1024, kSwizzle128);
            bool failed = false;
            auto proj = [&](int g) {
                wait_or_fail(fullx, g & 1, failed, status);
                tc_fence_after();
                constexpr uint32_t idU = idesc_bf16(64, C::NU, false, false);
#pragma unroll
                for (int kb = 0; kb < 2; ++kb)
#pragma unroll
                    for (int k = 0; k < 4; ++k) {
                        const uint64_t w = dadd(dW, kb * (C::NU * 128) + 32 * k);
                        mma_bf16_ss(tbase + cU, dadd(dQk, kb * T8 + 32 * k), w, idU, (kb | k) != 0);
                        mma_bf16_ss(tbase + cU + C::NU, dadd(dKk, kb * T8 + 32 * k), w, idU, (kb | k) != 0);
                    }
                mma_commit(uready);
            };
            if (T > 0) proj(0);
            Cursor64 cur;
            cur.start(a, it, false);
            for (int g = 0; g < T && !failed; ++g, cur.next(a, it)) {
                const int tin = cur.t;  // tile index within the item (z restarts at 0)
                wait_or_fail(phiready, g & 1, failed, status);
                wait_or_fail(fullvo, g & 1, failed, status);
                wait_or_fail(sopready, g & 1, failed, status);
                tc_fence_after();
                {
                    constexpr uint32_t idF = idesc_bf16(64, 64, false, false);
                    constexpr uint32_t idZc = idesc_bf16(64, C::D, false, true);
                    constexpr uint32_t idP = idesc_bf16(64, C::D, false, false);
#pragma unroll
                    for (int kb = 0; kb < 2; ++kb)
#pragma unroll
                        for (int k = 0; k < 4; ++k)
                            mma_bf16_ss(tbase + cU, dadd(dOk, kb * T8 + 32 * k), dadd(dVk, kb * T8 + 32 * k), idF,
                                        (kb | k) != 0);
#pragma unroll
                    for (int hl = 0; hl < 2; ++hl)
#pragma unroll
                        for (int k = 0; k < 4; ++k)
                            mma_bf16_ss(tbase + cZc, dadd(dL1, 32 * k), dadd(hl ? dPm : dKm, 2048 * k), idZc, (hl | k) != 0);
                    mma_commit(aready);  // the workers mask F while P = dO S^T runs
#pragma unroll
                    for (int h = 0; h < 2; ++h)
#pragma unroll
                        for (int kb = 0; kb < 2; ++kb)
#pragma unroll
                            for (int k = 0; k < 4; ++k)
                                mma_bf16_ss(tbase + cP, dadd(dOk, kb * T8 + 32 * k),
                                            dadd(h ? dSl : dSh, kb * C::T16 + 32 * k), idP, (h | kb | k) != 0);
                }
                wait_or_fail(fready, g & 1, failed, status);
                tc_fence_after();
                {
                    constexpr uint32_t idPi = idesc_bf16(64, C::D, false, true);
#pragma unroll
                    for (int k = 0; k < 4; ++k) {  // [F_hi, F_hi, F_lo] x [phi_hi, phi_lo, phi_hi]
                        mma_bf16_ss(tbase + cP, dadd(dFh, 32 * k), dadd(dKm, 2048 * k), idPi, 1u);
                        mma_bf16_ss(tbase + cP, dadd(dFh, 32 * k), dadd(dPm, 2048 * k), idPi, 1u);
                        mma_bf16_ss(tbase + cP, dadd(dFl, 32 * k), dadd(dKm, 2048 * k), idPi, 1u);
                    }
                    mma_commit(pready);
                    constexpr uint32_t idS = idesc_bf16(128, C::DV, true, true);
                    constexpr uint32_t idz = idesc_bf16(128, 16, true, false);
#pragma unroll
                    for (int hl = 0; hl < 2; ++hl)
#pragma unroll
                        for (int k = 0; k < 4; ++k) {
                            const uint64_t pa = dadd(hl ? dPm : dKm, 2048 * k);
                            mma_bf16_ss(tbase + cS, pa, dadd(dVm, 2048 * k), idS, 1u);
                            mma_bf16_ss(tbase + cz, pa, dadd(d1, 32 * k), idz, (tin > 0 || hl > 0 || k > 0) ? 1u : 0u);
                        }
                    mma_commit(sready);
                    mma_commit(infree);
                }
                if (g + 1 < T) proj(g + 1);  // U shares its columns with F, which the workers have read
            }
        }
    } else {
        const int q = warp & 3, cg = warp >> 2, h = lane >> 4;
        const int r = 16 * q + (lane & 15);           // row of the 64-row tile
        const int part = 2 * cg + h;                  // this thread's 16 features / columns: 16 * part ..
        const uint32_t lq = (uint32_t)(32 * q) << 16;  // TMEM lane base of the warp
        bool failed = false;
        float tq[TSUM ? 8 : 1] = {};  // channel normalisation: sums of phi . dphi per channel
        int g = 0;
        for (int item = it.begin; item < it.end; ++item) {
            const ItemRange ir = item_range(a, it, item);
            const int nt = tiles64(ir);
            if (nt == 0) continue;
            // segment start: S (TMEM fp32 and the bf16 hi/lo operand) and z from the prefix state
            {
                const float *Sp = a.seg_S + (head_state(a, ir.bh) * (a.nseg + 1) + ir.chunk) * C::D * C::DV;
                const int f = 32 * q + lane, c0 = 32 * cg;
                float v[32];
#pragma unroll
                for (int c = 0; c < 32; c += 4) {
                    const float4 x = __ldcg(reinterpret_cast<const float4 *>(Sp + (size_t)f * C::DV + c0 + c));
                    v[c] = x.x; v[c + 1] = x.y; v[c + 2] = x.z; v[c + 3] = x.w;
                }
                uint32_t w0[16], w1[16];
#pragma unroll
                for (int c = 0; c < 16; ++c) { w0[c] = __float_as_uint(v[c]); w1[c] = __float_as_uint(v[16 + c]); }
                tmem_st16(tbase + lq + cS + c0, w0);
                tmem_st16(tbase + lq + cS + c0 + 16, w1);
                tmem_wait_st();
                store_state32(Sh, Sl, f, c0, v);
                if (cg == 0) {
                    const float zv = __ldcg(a.seg_z + (head_state(a, ir.bh) * (a.nseg + 1) + ir.chunk) * C::D + f);
                    zpre[f] = zv;
                    sz[f] = zv;
                }
                fence_proxy_async_smem();
                tc_fence_before();
                mbar_arrive(sopready);
                named_sync<kCBWorkers>(1);
            }
            const size_t hrow = (size_t)ir.bh * a.n;  // workspace rows (staged rows, row statistics)
            for (int t = 0; t < nt; ++t, ++g) {
                const int row0 = ir.r0 + 64 * t;
                const int nvalid = min(64, ir.r1 - row0);
                const bool valid = r < nvalid;
                // A: phi(q) (fp32, kept), phi(k) (bf16 tile and global copy)
                wait_or_fail(uready, g & 1, failed, status);
                tc_fence_after();
                float phq[16];
                {
                    uint32_t x[4][4];
#pragma unroll
                    for (int s = 0; s < 4; ++s) tmem_ld4(tbase + lq + cU + 16 * s + 4 * cg, x[s]);
                    tmem_wait_ld();
                    float uu[4][2];  // [q hi, q mid, k hi, k mid][projection]
#pragma unroll
                    for (int s = 0; s < 4; ++s) {
                        const uint32_t xx[4] = {x[s][0], x[s][1], x[s][2], x[s][3]};
                        half_cols<2>(xx, uu[s], lane);
                    }
                    const int m0 = 4 * cg + 2 * h;
                    float u[4];
                    u[0] = uu[0][0] + uu[1][0] + sbias[m0];
                    u[1] = uu[0][1] + uu[1][1] + sbias[m0 + 1];
                    u[2] = uu[2][0] + uu[3][0] + sbias[m0];
                    u[3] = uu[2][1] + uu[3][1] + sbias[m0 + 1];
                    int node[4];
                    search_bucketed<4>(sTe, u, node);
                    const float4 *ab = reinterpret_cast<const float4 *>(sAB);
                    const float fl = channel_floor(a.lay);
                    float yk[16];
#pragma unroll
                    for (int p = 0; p < 4; ++p) {
                        const int jv = node[p];
#pragma unroll
                        for (int k = 0; k < 4; ++k) {
                            const float4 w = ab[ab_slot(jv, k)];
                            const float y0 = valid ? fmaxf(fmaf(w.x, u[p], w.y), fl) : 0.0f;
                            const float y1 = valid ? fmaxf(fmaf(w.z, u[p], w.w), fl) : 0.0f;
                            if (p < 2) { phq[8 * p + 2 * k] = y0; phq[8 * p + 2 * k + 1] = y1; }
                            else { yk[8 * (p - 2) + 2 * k] = y0; yk[8 * (p - 2) + 2 * k + 1] = y1; }
                        }
                    }
                    uint4 kh0, kl0, kh1, kl1;
                    {
                        const float y0[8] = {yk[0], yk[1], yk[2], yk[3], yk[4], yk[5], yk[6], yk[7]};
                        const float y1[8] = {yk[8], yk[9], yk[10], yk[11], yk[12], yk[13], yk[14], yk[15]};
                        split8(y0, kh0, kl0);
                        split8(y1, kh1, kl1);
                    }
                    const uint32_t boff = (m0 / 8) * T8;
                    *reinterpret_cast<uint4 *>(Kb + boff + sw128_chunk(r, m0 % 8)) = kh0;
                    *reinterpret_cast<uint4 *>(Kb + boff + sw128_chunk(r, m0 % 8 + 1)) = kh1;
                    *reinterpret_cast<uint4 *>(Pk + boff + sw128_chunk(r, m0 % 8)) = kl0;
                    *reinterpret_cast<uint4 *>(Pk + boff + sw128_chunk(r, m0 % 8 + 1)) = kl1;
                    if (valid) {  // workspace rows (32-byte aligned): [hi | lo] of the D features
                        uint4 *dst = reinterpret_cast<uint4 *>(static_cast<__nv_bfloat16 *>(a.phik) +
                                                               (hrow + row0 + r) * 2 * C::D + 16 * part);
                        st_v8(dst, kh0, kh1);
                        st_v8(dst + C::D / 8, kl0, kl1);
                    }
                }
                if (!valid && part == 0) {  // padded keys: clear V so that no garbage enters S
                    wait_or_fail(fullvo, g & 1, failed, status);
#pragma unroll
                    for (int kb = 0; kb < 2; ++kb)
#pragma unroll
                        for (int c = 0; c < 8; ++c)
                            *reinterpret_cast<uint4 *>(Vb + kb * T8 + sw128_chunk(r, c)) = make_uint4(0, 0, 0, 0);
                }
                fence_proxy_async_smem();
                tc_fence_before();
                mbar_arrive(phiready);
                // B: z_i = z + Zc_i, den parts; F masked to j <= i as hi + lo
                wait_or_fail(aready, g & 1, failed, status);
                tc_fence_after();
                float zi[16];
                uint32_t xf[16];
                {
                    uint32_t x[32], x1[16];
                    tmem_ld16(tbase + lq + cZc + 32 * cg, x1);
                    tmem_ld16(tbase + lq + cZc + 32 * cg + 16, *reinterpret_cast<uint32_t (*)[16]>(x + 16));
                    tmem_ld16(tbase + lq + cU + 16 * cg, xf);
                    tmem_wait_ld();
#pragma unroll
                    for (int k = 0; k < 16; ++k) x[k] = x1[k];
                    float zc[16];
                    half_cols<16>(x, zc, lane);
                    float dpart = 0.0f;
#pragma unroll
                    for (int k = 0; k < 16; ++k) {
                        zi[k] = sz[16 * part + k] + zc[k];
                        dpart = fmaf(phq[k], zi[k], dpart);
                    }
                    sred[part * 64 + r] = dpart;
                }
                {
                    float fv[8];
                    half_cols<8>(xf, fv, lane);
                    const int j0 = 8 * part;
#pragma unroll
                    for (int k = 0; k < 8; ++k) fv[k] = (valid && j0 + k <= r) ? fv[k] : 0.0f;
                    uint4 fh, fl;
                    split8(fv, fh, fl);
                    *reinterpret_cast<uint4 *>(Fh + sw128_chunk(r, part)) = fh;
                    *reinterpret_cast<uint4 *>(Fl + sw128_chunk(r, part)) = fl;
                }
                fence_proxy_async_smem();
                tc_fence_before();
                mbar_arrive(fready);
                // C: P -> ndot, dphi(q), phi~(q)
                wait_or_fail(pready, g & 1, failed, status);
                tc_fence_after();
                float pv[16];
                {
                    uint32_t x[32];
                    ld32(tbase + lq + cP + 32 * cg, x);
                    half_cols<16>(x, pv, lane);
                    float dot = 0.0f;
#pragma unroll
                    for (int k = 0; k < 16; ++k) dot = fmaf(phq[k], pv[k], dot);
                    sred[512 + part * 64 + r] = dot;
                }
                named_sync<kCBWorkers>(1);
                {
                    float den = 0.0f, dot = 0.0f;
#pragma unroll
                    for (int p = 0; p < 8; ++p) { den += sred[p * 64 + r]; dot += sred[512 + p * 64 + r]; }
                    den += a.eps;
                    const bool live = valid && den != 0.0f;
                    const float inv = live ? 1.0f / den : 0.0f;
                    const float ndot = -dot * inv;
                    float dq[16], pt[16];
#pragma unroll
                    for (int k = 0; k < 16; ++k) {
                        dq[k] = live ? (pv[k] + zi[k] * ndot) * inv : 0.0f;
                        pt[k] = phq[k] * inv;
                    }
                    if constexpr (TSUM) {  // feature 16 * part + k is channel k % 8
#pragma unroll
                        for (int k = 0; k < 16; ++k) tq[k & 7] = fmaf(phq[k], dq[k], tq[k & 7]);
                    }
                    if (valid) {  // workspace rows, 32-byte aligned
                        float4 *dst = reinterpret_cast<float4 *>(a.dphi + (hrow + row0 + r) * C::D + 16 * part);
#pragma unroll
                        for (int k = 0; k < 2; ++k)
                            st_v8(dst + 2 * k, f4_bits(make_float4(dq[8 * k], dq[8 * k + 1], dq[8 * k + 2], dq[8 * k + 3])),
                                  f4_bits(make_float4(dq[8 * k + 4], dq[8 * k + 5], dq[8 * k + 6], dq[8 * k + 7])));
                        uint4 h0, l0, h1, l1;
                        const float p0[8] = {pt[0], pt[1], pt[2], pt[3], pt[4], pt[5], pt[6], pt[7]};
                        const float p1[8] = {pt[8], pt[9], pt[10], pt[11], pt[12], pt[13], pt[14], pt[15]};
                        split8(p0, h0, l0);
                        split8(p1, h1, l1);
                        uint4 *pq = reinterpret_cast<uint4 *>(static_cast<__nv_bfloat16 *>(a.pq2) +
                                                              (hrow + row0 + r) * 2 * C::D + 16 * part);
                        st_v8(pq, h0, h1);
                        st_v8(pq + C::D / 8, l0, l1);
                        if (part == 0)
                            *reinterpret_cast<float2 *>(a.rowstat + 2 * (hrow + row0 + r)) =
                                make_float2(live ? den : 1.0f, live ? ndot : 0.0f);
                    }
                }
                // D: S after this tile -> operand of the next tile; z -> sz
                wait_or_fail(sready, g & 1, failed, status);
                tc_fence_after();
                if (t + 1 < nt) {
                    const int f = 32 * q + lane, c0 = 32 * cg;
                    uint32_t x[32];
                    ld32(tbase + lq + cS + c0, x);
                    float v[32];
#pragma unroll
                    for (int c = 0; c < 32; ++c) v[c] = __uint_as_float(x[c]);
                    store_state32(Sh, Sl, f, c0, v);
                    if (cg == 0) {
                        uint32_t zx[2];
                        tmem_ld2(tbase + lq + cz, zx);
                        tmem_wait_ld();
                        sz[f] = zpre[f] + __uint_as_float(zx[0]);
                    }
                    fence_proxy_async_smem();
                    tc_fence_before();
                    mbar_arrive(sopready);
                }
                named_sync<kCBWorkers>(1);  // sz, and sred free for the next tile
            }
        }
        if constexpr (TSUM) {  // the block's row of T: warp sums, then fp64 adds (the launch cleared the row)
#pragma unroll
            for (int l = 0; l < 8; ++l) {
                float v = tq[l];
#pragma unroll
                for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
                if (lane == 0) atomicAdd(tpart + (size_t)blockIdx.x * 8 + l, (double)v);
            }
        }
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 0) tmem_dealloc(tbase, 512);
}

// ---------------------------------------------------------------------------
// 2. segment sums of phi~(q) dO^T and phi~(q) ndot (128-row tiles)

constexpr int kSThreads = 192;  // warp 0: TMA, warp 1: MMA, warps 2-5: operand fixes and epilogue

template <class C>
__global__ void __launch_bounds__(kSThreads, 1)
    k_tcc_dstats(const __grid_constant__ CUtensorMap mapPq, const __grid_constant__ CUtensorMap mapdO, AttnArgs a,
                 int *status) {
    extern __shared__ uint8_t smem_raw[];
    uint8_t *sm = align1024(smem_raw);
    constexpr uint32_t T16 = C::T16;
    constexpr uint32_t STAGE = 4 * T16 + 2 * T16 + 4096;  // phi~ (hi, lo), dO, [ndot hi, lo] operand
    uint8_t *st = sm;                                      // [2] stages
    uint64_t *bars = reinterpret_cast<uint64_t *>(st + 2 * STAGE);
    uint64_t *full = bars, *fixed = bars + 2, *sfree = bars + 4, *accdone = bars + 6, *accfree = bars + 8;
    uint32_t *tslot = reinterpret_cast<uint32_t *>(bars + 10);
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const Items it(a);

    if (tid == 0) {
        for (int i = 0; i < 2; ++i) {
            mbar_init(full + i, 1); mbar_init(fixed + i, 128); mbar_init(sfree + i, 1);
            mbar_init(accdone + i, 1); mbar_init(accfree + i, 128);
        }
        fence_mbar_init();
    }
    if (warp == 0) { tmem_alloc(tslot, 512); tmem_relinquish(); }
    for (int e = tid; e < 2 * 4096 / 16; e += blockDim.x) {  // ndot operands: rows 2..15 stay zero
        const int s = e / 256, k = e % 256;
        reinterpret_cast<uint4 *>(st + s * STAGE + 6 * T16)[k] = make_uint4(0, 0, 0, 0);
    }
    fence_proxy_async_smem();
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tbase = *tslot;
    const int T = block_tiles(a, it);

    if (warp == 0) {
        if (lane == 0) {
            TileCursor cur;
            cur.start(a, it);
            bool failed = false;
            for (int g = 0; g < T && !failed; ++g, cur.next(a, it)) {
                const int s = g & 1;
                if (g >= 2) wait_or_fail(sfree + s, ((g - 2) >> 1) & 1, failed, status);
                mbar_arrive_expect_tx(full + s, 6 * T16);
                uint8_t *b = st + s * STAGE;
                for (int kb = 0; kb < 4; ++kb) tma_load_3d(b + kb * T16, &mapPq, kb * 64, cur.row0(), cur.g.bh, full + s);
                for (int kb = 0; kb < 2; ++kb)
                    tma_load_3d(b + (4 + kb) * T16, &mapdO, kb * 64, cur.row0(), cur.g.bh, full + s);
                if (g + 2 < T) {  // the tile after the next into L2 (two stages are in flight)
                    TileCursor nx = cur;
                    nx.next(a, it);
                    nx.next(a, it);
                    for (int kb = 0; kb < 4; ++kb) tma_prefetch_3d(&mapPq, kb * 64, nx.row0(), nx.g.bh);
                    for (int kb = 0; kb < 2; ++kb) tma_prefetch_3d(&mapdO, kb * 64, nx.row0(), nx.g.bh);
                }
            }
        }
    } else if (warp == 1) {
        if (lane == 0) {
            bool failed = false;
            int g = 0, ne = 0;
            for (int item = it.begin; item < it.end && !failed; ++item) {
                const int nt = item_range(a, it, item).ntiles;
                if (nt == 0) continue;
                const int b = ne & 1;
                if (ne >= 2) wait_or_fail(accfree + b, ((ne - 2) >> 1) & 1, failed, status);
                const uint32_t cS = tbase + b * 256, cZ = cS + 128;
                for (int t = 0; t < nt && !failed; ++t, ++g) {
                    const int s = g & 1;
                    wait_or_fail(fixed + s, (g >> 1) & 1, failed, status);
                    tc_fence_after();
                    const uint32_t base = smem_u32(st + s * STAGE);
                    const uint64_t dPm = sdesc(base, T16, 1024, kSwizzle128);            // MN-major, M = features
                    const uint64_t dOm = sdesc(base + 4 * T16, T16, 1024, kSwizzle128);  // MN-major, N = values
                    const uint64_t dN = sdesc(base + 6 * T16, 16, 1024, kSwizzle128);    // K-major, 16 rows
                    constexpr uint32_t idS = idesc_bf16(128, C::DV, true, true);
                    constexpr uint32_t idZ = idesc_bf16(128, 16, true, false);
#pragma unroll
                    for (int hl = 0; hl < 2; ++hl)
#pragma unroll
                        for (int k = 0; k < 8; ++k) {
                            const uint64_t pa = dadd(dPm, hl * 2 * T16 + 2048 * k);
                            mma_bf16_ss(cS, pa, dadd(dOm, 2048 * k), idS, (t | hl | k) != 0);
                            mma_bf16_ss(cZ, pa, dadd(dN, (k / 4) * 2048 + 32 * (k % 4)), idZ, (t | hl | k) != 0);
                        }
                    mma_commit(sfree + s);
                }
                mma_commit(accdone + b);
                ++ne;
            }
        }
    } else {
        const int ht = tid - 64;  // 0..127: key row of a tile; TMEM lane of the epilogue
        const uint32_t lrow = (uint32_t)((warp & 3) << 5) << 16;
        const int f = ((warp & 3) << 5) | lane;
        bool failed = false;
        int g = 0, ne = 0;
        for (int item = it.begin; item < it.end; ++item) {
            const ItemRange ir = item_range(a, it, item);
            for (int t = 0; t < ir.ntiles; ++t, ++g) {
                const int s = g & 1;
                const int row0 = ir.r0 + 128 * t;
                const bool valid = ht < min(128, ir.r1 - row0);
                wait_or_fail(full + s, (g >> 1) & 1, failed, status);
                uint8_t *b = st + s * STAGE;
                float nd = 0.0f;
                if (valid) nd = __ldcg(a.rowstat + 2 * ((size_t)ir.bh * a.n + row0 + ht) + 1);
                else {  // padded query rows: no garbage from dO
#pragma unroll
                    for (int kb = 0; kb < 2; ++kb)
#pragma unroll
                        for (int c = 0; c < 8; ++c)
                            *reinterpret_cast<uint4 *>(b + (4 + kb) * T16 + sw128_chunk(ht, c)) = make_uint4(0, 0, 0, 0);
                }
                __nv_bfloat16 hi, lo;
                split_bf16(nd, hi, lo);
                uint8_t *nb = b + 6 * T16 + (ht / 64) * 2048;
                *reinterpret_cast<__nv_bfloat16 *>(nb + sw128_chunk(0, (ht % 64) / 8) + (ht % 8) * 2) = hi;
                *reinterpret_cast<__nv_bfloat16 *>(nb + sw128_chunk(1, (ht % 64) / 8) + (ht % 8) * 2) = lo;
                fence_proxy_async_smem();
                mbar_arrive(fixed + s);
            }
            // epilogue of the item: its sums (zero for an item without tiles)
            float *Sp = a.dS_part + (size_t)item * C::D * C::DV;
            float *zp = a.dz_part + (size_t)item * C::D;
            if (ir.ntiles == 0) {
                for (int c = 0; c < C::DV; c += 4)
                    *reinterpret_cast<float4 *>(Sp + (size_t)f * C::DV + c) = make_float4(0.f, 0.f, 0.f, 0.f);
                zp[f] = 0.0f;
                continue;
            }
            const int bsel = ne & 1;
            wait_or_fail(accdone + bsel, (ne >> 1) & 1, failed, status);
            tc_fence_after();
            const uint32_t cS = tbase + lrow + bsel * 256;
#pragma unroll
            for (int c0 = 0; c0 < C::DV; c0 += 32) {
                uint32_t x[32];
                ld32(cS + c0, x);
#pragma unroll
                for (int c = 0; c < 32; c += 4)
                    *reinterpret_cast<float4 *>(Sp + (size_t)f * C::DV + c0 + c) =
                        make_float4(__uint_as_float(x[c]), __uint_as_float(x[c + 1]), __uint_as_float(x[c + 2]),
                                    __uint_as_float(x[c + 3]));
            }
            uint32_t zx[2];
            tmem_ld2(cS + 128, zx);
            tmem_wait_ld();
            zp[f] = __uint_as_float(zx[0]) + __uint_as_float(zx[1]);
            tc_fence_before();
            mbar_arrive(accfree + bsel);
            ++ne;
        }
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 0) tmem_dealloc(tbase, 512);
}

// ---------------------------------------------------------------------------
// 3. exclusive suffix over the segments: seg_dS[bh][s] = sum_{s' > s} dS_part[bh][s']

__global__ void __launch_bounds__(256) k_seg_rscan(AttnArgs a) {
    const int bh = blockIdx.y;
    const size_t SD = (size_t)a.D * a.dv;
    const int e4 = blockIdx.x * blockDim.x + threadIdx.x;
    if ((size_t)e4 * 4 < SD) {
        const float4 *part = reinterpret_cast<const float4 *>(a.dS_part + (size_t)bh * a.nseg * SD) + e4;
        float4 *out = reinterpret_cast<float4 *>(a.seg_dS + (size_t)bh * a.nseg * SD) + e4;
        float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
        for (int s = a.nseg - 1; s >= 0; --s) {
            const float4 v = __ldcg(part + (size_t)s * (SD / 4));
            out[(size_t)s * (SD / 4)] = acc;
            acc.x += v.x; acc.y += v.y; acc.z += v.z; acc.w += v.w;
        }
    }
    if (blockIdx.x == 0) {
        for (int f = threadIdx.x; f < a.D; f += blockDim.x) {
            const float *part = a.dz_part + (size_t)bh * a.nseg * a.D + f;
            float *out = a.seg_dz + (size_t)bh * a.nseg * a.D + f;
            float acc = 0.0f;
            for (int s = a.nseg - 1; s >= 0; --s) {
                const float v = __ldcg(part + (size_t)s * a.D);
                out[(size_t)s * a.D] = acc;
                acc += v;
            }
        }
    }
}

// ---------------------------------------------------------------------------
// 4. key side (reverse sweep)

template <class C>
__global__ void __launch_bounds__(kCBThreads, 1)
    k_tcc_key(const __grid_constant__ CUtensorMap mapPk, const __grid_constant__ CUtensorMap mapPq,
              const __grid_constant__ CUtensorMap mapV, const __grid_constant__ CUtensorMap mapdO, AttnArgs a,
              int *status) {
    extern __shared__ uint8_t smem_raw[];
    uint8_t *sm = align1024(smem_raw);
    constexpr uint32_t T8 = C::T8, RT = C::RT;
    uint8_t *Pk = sm;                // phi(K): hi blocks 0, 1; lo blocks 2, 3 ([key][feature])
    uint8_t *Pq = Pk + 2 * RT;       // phi~(Q): hi blocks 0, 1; lo blocks 2, 3 ([query][feature])
    uint8_t *Vb = Pq + 2 * RT;
    uint8_t *Ob = Vb + RT;           // dO
    uint8_t *Nd = Ob + RT;           // [ndot hi, ndot lo, 0...] x 64 queries (K-major, 16 rows)
    uint8_t *Ch = Nd + 2048;         // masked C, hi and lo [key][query]
    uint8_t *Cl = Ch + T8;
    uint8_t *Eh = Cl + T8;           // masked E + ndot, hi and lo [key][query]
    uint8_t *El = Eh + T8;
    uint8_t *Sh = El + T8;           // dS operand [feature][value], hi and lo
    uint8_t *Sl = Sh + C::SOP;
    float *sdz = reinterpret_cast<float *>(Sl + C::SOP);
    uint64_t *bars = reinterpret_cast<uint64_t *>(sdz + C::D);
    uint64_t *full = bars, *infree = bars + 1, *c1ready = bars + 2, *mready = bars + 3;
    uint64_t *c3ready = bars + 4, *accfree = bars + 5, *sopready = bars + 6;
    uint64_t *dvready = bars + 7, *dfready = bars + 8;
    uint32_t *tslot = reinterpret_cast<uint32_t *>(bars + 9);

    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const Items it(a);
    // TMEM: dV (C first) [128] | dphi (E first) [128] | dS [128] | dz [16]
    constexpr uint32_t cV = 0, cF = 128, cS = 256, cZ = 384;

    if (tid == 0) {
        mbar_init(full, 1); mbar_init(infree, 1); mbar_init(c1ready, 1); mbar_init(mready, kCBWorkers);
        mbar_init(c3ready, 1); mbar_init(accfree, kCBWorkers); mbar_init(sopready, kCBWorkers);
        mbar_init(dvready, 1); mbar_init(dfready, 1);
        fence_mbar_init();
    }
    if (warp == 0) { tmem_alloc(tslot, 512); tmem_relinquish(); }
    for (int e = tid; e < 2048 / 16; e += blockDim.x) reinterpret_cast<uint4 *>(Nd)[e] = make_uint4(0, 0, 0, 0);
    // rows beyond the sequence length receive zero dV
    for (int item = it.begin; item < it.end; ++item) {
        const ItemRange ir = item_range(a, it, item);
        __nv_bfloat16 *dV = static_cast<__nv_bfloat16 *>(a.dV) + head_rows(a, ir.bh) * C::DV;
        const int z0 = max(ir.r0, ir.r1);
        for (int e = tid; e < (ir.rend - z0) * C::DV / 8; e += blockDim.x)
            reinterpret_cast<uint4 *>(dV + (size_t)z0 * C::DV)[e] = make_uint4(0, 0, 0, 0);
    }
    fence_proxy_async_smem();
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tbase = *tslot;
    const int T = block_tiles64(a, it);

    if (warp == kCBTma) {
        if (lane == 0) {
            Cursor64 cur;
            cur.start(a, it, true);
            bool failed = false;
            for (int g = 0; g < T && !failed; ++g, cur.next(a, it)) {
                if (g >= 1) wait_or_fail(infree, (g - 1) & 1, failed, status);
                mbar_arrive_expect_tx(full, 6 * RT);
                const int r0 = cur.row0(), bh = cur.g.bh;
                for (int kb = 0; kb < 2; ++kb) {
                    tma_load_3d(Vb + kb * T8, &mapV, kb * 64, r0, bh, full);
                    tma_load_3d(Ob + kb * T8, &mapdO, kb * 64, r0, bh, full);
                }
                for (int kb = 0; kb < 4; ++kb) {
                    tma_load_3d(Pk + kb * T8, &mapPk, kb * 64, r0, bh, full);
                    tma_load_3d(Pq + kb * T8, &mapPq, kb * 64, r0, bh, full);
                }
                if (g + 1 < T && !failed) {  // the next tile into L2 while this one is worked on
                    Cursor64 nx = cur;
                    nx.next(a, it);
                    const int n0 = nx.row0(), nb = nx.g.bh;
                    for (int kb = 0; kb < 2; ++kb) {
                        tma_prefetch_3d(&mapV, kb * 64, n0, nb);
                        tma_prefetch_3d(&mapdO, kb * 64, n0, nb);
                    }
                    for (int kb = 0; kb < 4; ++kb) {
                        tma_prefetch_3d(&mapPk, kb * 64, n0, nb);
                        tma_prefetch_3d(&mapPq, kb * 64, n0, nb);
                    }
                }
            }
        }
    } else if (warp == kCBMma) {
        if (lane == 0) {
            const uint64_t dPkK = sdesc(smem_u32(Pk), 16, 1024, kSwizzle128);   // K-major, rows = keys
            const uint64_t dPqK = sdesc(smem_u32(Pq), 16, 1024, kSwizzle128);   // K-major, rows = queries
            const uint64_t dPqM = sdesc(smem_u32(Pq), T8, 1024, kSwizzle128);   // MN-major, M/N = features
            const uint64_t dVk = sdesc(smem_u32(Vb), 16, 1024, kSwizzle128);
            const uint64_t dOk = sdesc(smem_u32(Ob), 16, 1024, kSwizzle128);
            const uint64_t dOm = sdesc(smem_u32(Ob), T8, 1024, kSwizzle128);    // MN-major, N = values
            const uint64_t dN = sdesc(smem_u32(Nd), 16, 1024, kSwizzle128);
            const uint64_t dCh = sdesc(smem_u32(Ch), 16, 1024, kSwizzle128);
            const uint64_t dCl = sdesc(smem_u32(Cl), 16, 1024, kSwizzle128);
            const uint64_t dEh = sdesc(smem_u32(Eh), 16, 1024, kSwizzle128);
            const uint64_t dEl = sdesc(smem_u32(El), 16, 1024, kSwizzle128);
            const uint64_t dShM = sdesc(smem_u32(Sh), C::T16, 1024, kSwizzle128);  // MN-major, N = values
            const uint64_t dSlM = sdesc(smem_u32(Sl), C::T16, 1024, kSwizzle128);
            const uint64_t dShK = sdesc(smem_u32(Sh), 16, 1024, kSwizzle128);      // K-major, rows = features
            const uint64_t dSlK = sdesc(smem_u32(Sl), 16, 1024, kSwizzle128);
            bool failed = false;
            for (int g = 0; g < T && !failed; ++g) {
                // C = phi(K) phi~(Q)^T ([hi, hi, lo] x [hi, lo, hi]), E = V dO^T
                wait_or_fail(full, g & 1, failed, status);
                if (g >= 1) wait_or_fail(accfree, (g - 1) & 1, failed, status);
                tc_fence_after();
                {
                    constexpr uint32_t id64 = idesc_bf16(64, 64, false, false);
#pragma unroll
                    for (int kb = 0; kb < 2; ++kb)
#pragma unroll
                        for (int k = 0; k < 4; ++k) {
                            const uint32_t o = kb * T8 + 32 * k;
                            mma_bf16_ss(tbase + cV, dadd(dPkK, o), dadd(dPqK, o), id64, (kb | k) != 0);
                            mma_bf16_ss(tbase + cV, dadd(dPkK, o), dadd(dPqK, 2 * T8 + o), id64, 1u);
                            mma_bf16_ss(tbase + cV, dadd(dPkK, 2 * T8 + o), dadd(dPqK, o), id64, 1u);
                            mma_bf16_ss(tbase + cF, dadd(dVk, o), dadd(dOk, o), id64, (kb | k) != 0);
                        }
                    mma_commit(c1ready);
                }
                wait_or_fail(mready, g & 1, failed, status);
                wait_or_fail(sopready, g & 1, failed, status);
                tc_fence_after();
                {
                    // dV = phi(K) dS ([hi, hi, lo] x [hi, lo, hi]) + C dO (C hi + lo)
                    constexpr uint32_t idV = idesc_bf16(64, C::DV, false, true);
#pragma unroll
                    for (int kb = 0; kb < 2; ++kb)
#pragma unroll
                        for (int k = 0; k < 4; ++k) {
                            const uint32_t o = kb * T8 + 32 * k, so = (4 * kb + k) * 2048;
                            mma_bf16_ss(tbase + cV, dadd(dPkK, o), dadd(dShM, so), idV, (kb | k) != 0);
                            mma_bf16_ss(tbase + cV, dadd(dPkK, o), dadd(dSlM, so), idV, 1u);
                            mma_bf16_ss(tbase + cV, dadd(dPkK, 2 * T8 + o), dadd(dShM, so), idV, 1u);
                        }
#pragma unroll
                    for (int k = 0; k < 4; ++k) {
                        mma_bf16_ss(tbase + cV, dadd(dCh, 32 * k), dadd(dOm, 2048 * k), idV, 1u);
                        mma_bf16_ss(tbase + cV, dadd(dCl, 32 * k), dadd(dOm, 2048 * k), idV, 1u);
                    }
                    mma_commit(dvready);
                    // dphi = V [dS_hi; dS_lo]^T + E phi~(Q)   (E hi x phi~ hi, lo; E lo x phi~ hi)
                    constexpr uint32_t idF = idesc_bf16(64, C::D, false, false);
                    constexpr uint32_t idFm = idesc_bf16(64, C::D, false, true);
#pragma unroll
                    for (int hl = 0; hl < 2; ++hl)
#pragma unroll
                        for (int kb = 0; kb < 2; ++kb)
#pragma unroll
                            for (int k = 0; k < 4; ++k)
                                mma_bf16_ss(tbase + cF, dadd(dVk, kb * T8 + 32 * k),
                                            dadd(hl ? dSlK : dShK, kb * C::T16 + 32 * k), idF, (hl | kb | k) != 0);
#pragma unroll
                    for (int k = 0; k < 4; ++k) {
                        mma_bf16_ss(tbase + cF, dadd(dEh, 32 * k), dadd(dPqM, 2048 * k), idFm, 1u);
                        mma_bf16_ss(tbase + cF, dadd(dEh, 32 * k), dadd(dPqM, 2 * T8 + 2048 * k), idFm, 1u);
                        mma_bf16_ss(tbase + cF, dadd(dEl, 32 * k), dadd(dPqM, 2048 * k), idFm, 1u);
                    }
                    mma_commit(dfready);
                    // dS += phi~(Q)^T dO, dz += phi~(Q)^T [ndot_hi, ndot_lo]
                    constexpr uint32_t idS = idesc_bf16(128, C::DV, true, true);
                    constexpr uint32_t idZ = idesc_bf16(128, 16, true, false);
#pragma unroll
                    for (int hl = 0; hl < 2; ++hl)
#pragma unroll
                        for (int k = 0; k < 4; ++k) {
                            const uint64_t pa = dadd(dPqM, hl * 2 * T8 + 2048 * k);
                            mma_bf16_ss(tbase + cS, pa, dadd(dOm, 2048 * k), idS, 1u);
                            mma_bf16_ss(tbase + cZ, pa, dadd(dN, 32 * k), idZ, 1u);
                        }
                    mma_commit(c3ready);
                    mma_commit(infree);
                }
            }
        }
    } else {
        const int q = warp & 3, cg = warp >> 2, h = lane >> 4;
        const int r = 16 * q + (lane & 15);           // key row of the 64-row tile
        const int part = 2 * cg + h;
        const uint32_t lq = (uint32_t)(32 * q) << 16;
        bool failed = false;
        int g = 0;
        for (int item = it.begin; item < it.end; ++item) {
            const ItemRange ir = item_range(a, it, item);
            const int nt = tiles64(ir);
            if (nt == 0) continue;
            // segment end: dS, dz after the segment (suffix of the later segments)
            {
                const float *Sp = a.seg_dS + ((size_t)ir.bh * a.nseg + ir.chunk) * C::D * C::DV;
                const int f = 32 * q + lane, c0 = 32 * cg;
                float v[32];
#pragma unroll
                for (int c = 0; c < 32; c += 4) {
                    const float4 x = __ldcg(reinterpret_cast<const float4 *>(Sp + (size_t)f * C::DV + c0 + c));
                    v[c] = x.x; v[c + 1] = x.y; v[c + 2] = x.z; v[c + 3] = x.w;
                }
                uint32_t w0[16], w1[16];
#pragma unroll
                for (int c = 0; c < 16; ++c) { w0[c] = __float_as_uint(v[c]); w1[c] = __float_as_uint(v[16 + c]); }
                tmem_st16(tbase + lq + cS + c0, w0);
                tmem_st16(tbase + lq + cS + c0 + 16, w1);
                store_state32(Sh, Sl, f, c0, v);
                if (cg == 0) {
                    const float zv = __ldcg(a.seg_dz + ((size_t)ir.bh * a.nseg + ir.chunk) * C::D + f);
                    uint32_t zw[16];
#pragma unroll
                    for (int c = 0; c < 16; ++c) zw[c] = 0u;
                    zw[0] = __float_as_uint(zv);
                    tmem_st16(tbase + lq + cZ, zw);
                    sdz[f] = zv;
                }
                tmem_wait_st();
                fence_proxy_async_smem();
                tc_fence_before();
                mbar_arrive(sopready);
                named_sync<kCBWorkers>(1);
            }
            const size_t hrow = (size_t)ir.bh * a.n;  // workspace rows (staged rows, row statistics)
            const size_t urow = head_rows(a, ir.bh);  // the caller's rows (dV)
            for (int tr = 0; tr < nt; ++tr, ++g) {
                const int t = nt - 1 - tr;
                const int row0 = ir.r0 + 64 * t;
                const int nvalid = min(64, ir.r1 - row0);
                const bool valid = r < nvalid;
                // masked C and E + ndot; padded query rows of dO cleared; ndot operand
                const int i0 = 8 * part;
                float nd[8], ndr = 0.0f;  // -dO.O of this thread's 8 query columns and of its own row
#pragma unroll
                for (int k = 0; k < 8; ++k)
                    nd[k] = (i0 + k < nvalid) ? __ldcg(a.rowstat + 2 * (hrow + row0 + i0 + k) + 1) : 0.0f;
                if (part == 0 && valid) ndr = __ldcg(a.rowstat + 2 * (hrow + row0 + r) + 1);
                wait_or_fail(c1ready, g & 1, failed, status);
                tc_fence_after();
                {
                    uint32_t x[16];
                    tmem_ld16(tbase + lq + cV + 16 * cg, x);
                    tmem_wait_ld();
                    float cv[8];
                    half_cols<8>(x, cv, lane);
                    tmem_ld16(tbase + lq + cF + 16 * cg, x);
                    tmem_wait_ld();
                    float ev[8];
                    half_cols<8>(x, ev, lane);
#pragma unroll
                    for (int k = 0; k < 8; ++k) {
                        const bool keep = valid && i0 + k >= r && i0 + k < nvalid;
                        cv[k] = keep ? cv[k] : 0.0f;
                        ev[k] = keep ? ev[k] + nd[k] : 0.0f;
                    }
                    uint4 ch, cl;
                    split8(cv, ch, cl);
                    *reinterpret_cast<uint4 *>(Ch + sw128_chunk(r, part)) = ch;
                    *reinterpret_cast<uint4 *>(Cl + sw128_chunk(r, part)) = cl;
                    uint4 eh, el;
                    split8(ev, eh, el);
                    *reinterpret_cast<uint4 *>(Eh + sw128_chunk(r, part)) = eh;
                    *reinterpret_cast<uint4 *>(El + sw128_chunk(r, part)) = el;
                }
                if (part == 0) {
                    if (!valid) {
#pragma unroll
                        for (int kb = 0; kb < 2; ++kb)
#pragma unroll
                            for (int c = 0; c < 8; ++c)
                                *reinterpret_cast<uint4 *>(Ob + kb * T8 + sw128_chunk(r, c)) = make_uint4(0, 0, 0, 0);
                    }
                    __nv_bfloat16 hi, lo;
                    split_bf16(ndr, hi, lo);
                    *reinterpret_cast<__nv_bfloat16 *>(Nd + sw128_chunk(0, r / 8) + (r % 8) * 2) = hi;
                    *reinterpret_cast<__nv_bfloat16 *>(Nd + sw128_chunk(1, r / 8) + (r % 8) * 2) = lo;
                }
                fence_proxy_async_smem();
                tc_fence_before();
                mbar_arrive(mready);
                // dV, dphi(k) = dphi + dz (the state after this tile's rows)
                wait_or_fail(dvready, g & 1, failed, status);
                tc_fence_after();
                {
                    uint32_t x[32];
                    ld32(tbase + lq + cV + 32 * cg, x);
                    float dv[16];
                    half_cols<16>(x, dv, lane);
                    if (valid) {
                        uint4 *dst = reinterpret_cast<uint4 *>(static_cast<__nv_bfloat16 *>(a.dV) +
                                                               (urow + row0 + r) * C::DV + 16 * part);
                        dst[0] = pack8f(dv);
                        dst[1] = pack8f(dv + 8);
                    }
                    wait_or_fail(dfready, g & 1, failed, status);
                    tc_fence_after();
                    ld32(tbase + lq + cF + 32 * cg, x);
                    float df[16];
                    half_cols<16>(x, df, lane);
                    tc_fence_before();
                    mbar_arrive(accfree);
                    if (valid) {  // workspace rows, 32-byte aligned
                        float4 *fp = reinterpret_cast<float4 *>(a.dphi + (hrow + row0 + r) * C::D + 16 * part);
                        float o[16];
#pragma unroll
                        for (int k = 0; k < 16; ++k) o[k] = df[k] + sdz[16 * part + k];
#pragma unroll
                        for (int k = 0; k < 2; ++k)
                            st_v8(fp + 2 * k, f4_bits(make_float4(o[8 * k], o[8 * k + 1], o[8 * k + 2], o[8 * k + 3])),
                                  f4_bits(make_float4(o[8 * k + 4], o[8 * k + 5], o[8 * k + 6], o[8 * k + 7])));
                    }
                }
                named_sync<kCBWorkers>(1);  // every sdz read before it changes
                wait_or_fail(c3ready, g & 1, failed, status);
                tc_fence_after();
                if (tr + 1 < nt) {  // dS, dz after this tile -> operand and sdz of the next (earlier) tile
                    const int f = 32 * q + lane, c0 = 32 * cg;
                    uint32_t x[32];
                    ld32(tbase + lq + cS + c0, x);
                    float v[32];
#pragma unroll
                    for (int c = 0; c < 32; ++c) v[c] = __uint_as_float(x[c]);
                    store_state32(Sh, Sl, f, c0, v);
                    if (cg == 0) {
                        uint32_t zx[2];
                        tmem_ld2(tbase + lq + cZ, zx);
                        tmem_wait_ld();
                        sdz[f] = __uint_as_float(zx[0]) + __uint_as_float(zx[1]);
                    }
                    fence_proxy_async_smem();
                    tc_fence_before();
                    mbar_arrive(sopready);
                }
                named_sync<kCBWorkers>(1);  // sdz of the next tile
            }
        }
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 0) tmem_dealloc(tbase, 512);
}

}  // namespace

bool tc_make_map_rows(CUtensorMap *m, const void *base, int width, int n, int BH, int rows, int hs_mul);
int tc_sm_count();
cudaError_t launch_tc_causal_stats(const AttnArgs &a, cudaStream_t s);
cudaError_t launch_tc_phi_bwd(const AttnArgs &a, const void *X, const float *dphi, void *dX, int slot0, int grid,
                              cudaStream_t s, const float *kfold = nullptr);

cudaError_t launch_tc_causal_bwd(const AttnArgs &a0, bool have_state, cudaStream_t s) {
    using C = K64;
    AttnArgs a = a0;
    a.rows_per_split = a0.seg_len;  // work item = state segment
    a.nsplit = a0.nseg;
    cudaError_t e;
    if (!have_state && (e = launch_tc_causal_stats(a, s)) != cudaSuccess) return e;
    const int BH = a.B * a.H;
    const int items = BH * a.nseg;
    const int grid = items < tc_sm_count() ? items : tc_sm_count();
    int *st = reinterpret_cast<int *>(reinterpret_cast<char *>(a.counters) - 256);
    CUtensorMap mQ, mK, mV, mdO, mPk, mPq, mPq128, mdO128;
    const int hm = a.hs_mul;  // the caller's tensors; the staged rows (phi(k), phi(q)/den) are the workspace's
    if (!tc_make_map_rows(&mQ, a.Q, a.d, a.n, BH, 64, hm) || !tc_make_map_rows(&mK, a.K, a.d, a.n, BH, 64, hm) ||
        !tc_make_map_rows(&mV, a.V, a.dv, a.n, BH, 64, hm) || !tc_make_map_rows(&mdO, a.dO, a.dv, a.n, BH, 64, hm) ||
        !tc_make_map_rows(&mPk, a.phik, 2 * C::D, a.n, BH, 64, 1) ||
        !tc_make_map_rows(&mPq, a.pq2, 2 * C::D, a.n, BH, 64, 1) ||
        !tc_make_map_rows(&mPq128, a.pq2, 2 * C::D, a.n, BH, 128, 1) ||
        !tc_make_map_rows(&mdO128, a.dO, a.dv, a.n, BH, 128, hm))
        return cudaErrorInvalidValue;
    // 1. query side
    if ((e = cudaFuncSetAttribute(k_tcc_query<C, false>, cudaFuncAttributeMaxDynamicSharedMemorySize, C::SMEM_Q)) !=
            cudaSuccess ||
        (e = cudaFuncSetAttribute(k_tcc_query<C, true>, cudaFuncAttributeMaxDynamicSharedMemorySize, C::SMEM_Q)) !=
            cudaSuccess)
        return e;
    // with the channel normalisation the sweep also sums phi^ . dphi^ per channel and block (T), so that
    // the scale term's kappa is known before either chain rule, which then adds M kappa_l phi^ to dphi^
    double *tpart = a.ch_sigma ? a.ch_T : nullptr;
    if (tpart && (e = cudaMemsetAsync(tpart, 0, (size_t)grid * 8 * sizeof(double), s)) != cudaSuccess) return e;
    if (tpart)
        LUNA_LAUNCH("tcc_query", (k_tcc_query<C, true>), grid, kCBThreads, C::SMEM_Q, s, mQ, mK, mV, mdO, a, tpart, st);
    else
        LUNA_LAUNCH("tcc_query", (k_tcc_query<C, false>), grid, kCBThreads, C::SMEM_Q, s, mQ, mK, mV, mdO, a, tpart, st);
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
    if (a.ch_sigma) {
        a.ch_T_rows = grid;
        if ((e = launch_chrms_kappa(a, s)) != cudaSuccess) return e;
    }
    const float *kq = a.ch_sigma ? a.ch_kappa : nullptr, *kk = a.ch_sigma ? a.ch_kappa + kMaxL : nullptr;
    if ((e = launch_tc_phi_bwd(a, a.Q, a.dphi, a.dQ, 0, grid, s, kq)) != cudaSuccess) return e;
    // 2, 3. segment sums of dS, dz and their suffix
    constexpr uint32_t SMEM_S = 2 * (6 * C::T16 + 4096) + 128 + 1024;
    static_assert(SMEM_S <= kSmemLimit, "shared memory budget");
    if ((e = cudaFuncSetAttribute(k_tcc_dstats<C>, cudaFuncAttributeMaxDynamicSharedMemorySize, SMEM_S)) != cudaSuccess)
        return e;
    LUNA_LAUNCH("tcc_dstats", k_tcc_dstats<C>, grid, kSThreads, SMEM_S, s, mPq128, mdO128, a, st);
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
    const size_t SD4 = (size_t)a.D * a.dv / 4;
    LUNA_LAUNCH("seg_rscan", k_seg_rscan, dim3((unsigned)((SD4 + 255) / 256), BH), 256, 0, s, a);
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
    // 4. key side
    if ((e = cudaFuncSetAttribute(k_tcc_key<C>, cudaFuncAttributeMaxDynamicSharedMemorySize, C::SMEM_K)) != cudaSuccess)
        return e;
    LUNA_LAUNCH("tcc_key", k_tcc_key<C>, grid, kCBThreads, C::SMEM_K, s, mPk, mPq, mV, mdO, a, st);
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
    // 5. chain rule for K, then the parameter-gradient reduction over both sides
    if ((e = launch_tc_phi_bwd(a, a.K, a.dphi, a.dK, grid, grid, s, kk)) != cudaSuccess) return e;
    return launch_grad_reduce(a, 2 * grid, s);
}

}  // namespace luna
