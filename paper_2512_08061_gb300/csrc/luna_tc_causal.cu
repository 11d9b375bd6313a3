// Streaming (causal) form of Eq. (kernel-attn) on tensor cores (bf16 I/O, sm_103a):
//     O_i = phi(q_i)^T S_i / (phi(q_i)^T z_i + eps),  S_i = sum_{j<=i} phi(k_j) v_j^T,  z_i = sum_{j<=i} phi(k_j).
//
// The rows of a head are cut into state segments (whole 128-row tiles).
//   1. Key statistics of every segment (the key-pass kernel in per-item mode).
//   2. k_seg_scan: exclusive prefix of those statistics at every segment start
//      (and the total), the state that the backward pass reads.
//   3. k_tc_causal: a persistent block walks its segments tile by tile and
//      keeps the running S (fp32) in TMEM.  Per 128-row tile, with S, z the
//      state before the tile:
//        MMA   U = [Q; K] W^T                       (projections)
//        work  phi(Q), phi(K) as bf16 tiles; fp32 phi(q) . z
//        MMA   num = phi(Q) S_bf16,  A = phi(Q) phi(K)^T
//        work  A masked to keys j <= i, its row sums, A as bf16
//        MMA   num += A V,  S += phi(K)^T V,  z += phi(K)^T 1
//        work  O = num / (phi(q).z + rowsum(A) + eps);  S -> bf16 operand of the next tile
//      The MMA warp issues the next tile's U_q (into a second TMEM slot) right
//      after num and A, so that the X buffer takes the next K tile while the
//      workers mask the scores, and the next U_k after the O products, while
//      the workers write O.
//      S, phi and the scores enter the products as one bf16 rounding (the
//      forward output is bf16; the backward pass recomputes its own state from
//      the exact segment prefixes of step 2).  The normaliser uses the same
//      rounded phi(q) and scores as the numerator, so that each output row
//      stays a normalised combination of the values.
#include "luna_tc_dev.cuh"

namespace luna {
namespace {
using namespace sm100;
using namespace simt;
using namespace tcdev;

constexpr int kCWorkers = 512;  // 16 warps, four threads per row
constexpr int kCTma = 16, kCMma = 17;
constexpr int kCThreads = kCWorkers + 64;

// d = dv = 128, M = 16 projections, L = 8 channels: D = 128 features
struct K128 {
    static constexpr int d = 128, DX = 128, DV = 128, MP = 16, D = 128, NU = 32, PP = 4;
    static constexpr int KBX = DX / 64;
    static constexpr uint32_t TILE = 16384;        // 128 rows x 128 B (one 64-column block)
    static constexpr uint32_t XT = 128 * DX * 2;   // Q or K tile
    static constexpr uint32_t VT = 128 * DV * 2;   // V tile
    static constexpr uint32_t PT = 128 * D * 2;    // phi tile; also the 128 x 128 score tile A
    static constexpr uint32_t ST = D * DV * 2;     // S operand, MN-major: [value block][feature][64 values]
    static constexpr uint32_t ONES = 16 * 128 * 2; // K-major ones operand: 16 rows x 128 keys
    static constexpr uint32_t WOP = NU * DX * 2;
    static constexpr uint32_t SMEM = XT + VT + 2 * PT + ST + ONES + WOP + kTableBytes + D * 4 * 2 + 4 * 128 * 4 +
                                     256 + 1024;
    static_assert(SMEM <= kSmemLimit, "shared memory budget");
    static_assert(PT == 2 * TILE && XT == 2 * TILE && VT == 2 * TILE && ST == 2 * TILE, "two 64-column blocks");
};

// TMEM columns: U (q of even tiles: 0..31, k: 32..63) | num | A | S | z | q of odd tiles
constexpr uint32_t cU = 0, cN = 64, cA = 192, cS = 320, cZ = 448, cUq1 = 464;
__host__ __device__ constexpr uint32_t col_uq(int g) { return (g & 1) ? cUq1 : cU; }

// phi of projections Qd*PP .. Qd*PP+PP-1 of one row of the Q tile and of the
// K tile, from their projection columns (hi at u, mid at u + MP): bf16 chunks
// into the phi tiles (zeros if !valid).  The 2 * PP interval searches run
// interleaved.  Returns the fp32 dot product of the bf16 phi(q) features with
// sz, the normaliser part that the numerator's rounding matches.
template <class C>
__device__ __forceinline__ float phi_quarter_qk(uint32_t uq, uint32_t uk, int Qd, const float *sTe, const float *sAB,
                                                const float *sbias, float fl, bool valid, int r, uint8_t *tq,
                                                uint8_t *tk, const float *sz) {
    constexpr int PP = C::PP;
    static_assert(PP == 4, "four projections per thread");
    float u[2 * PP];
    {
        uint32_t qh[4], qm[4], kh[4], km[4];
        tmem_ld4(uq + Qd * PP, qh);
        tmem_ld4(uq + C::MP + Qd * PP, qm);
        tmem_ld4(uk + Qd * PP, kh);
        tmem_ld4(uk + C::MP + Qd * PP, km);
        tmem_wait_ld();
#pragma unroll
        for (int q = 0; q < PP; ++q) {
            const float b = sbias[Qd * PP + q];
            u[q] = __uint_as_float(qh[q]) + __uint_as_float(qm[q]) + b;
            u[PP + q] = __uint_as_float(kh[q]) + __uint_as_float(km[q]) + b;
        }
    }
    int node[2 * PP];
    search_bucketed<2 * PP>(sTe, u, node);
    float dot = 0.0f;
    const float4 *ab = reinterpret_cast<const float4 *>(sAB);
#pragma unroll
    for (int q = 0; q < 2 * PP; ++q) {
        const int i = Qd * PP + (q % PP), j = node[q];
        uint4 w = make_uint4(0u, 0u, 0u, 0u);
        if (valid) {
            float y[8];
#pragma unroll
            for (int k = 0; k < 4; ++k) {
                const float4 v = ab[ab_slot(j, k)];
                y[2 * k] = fmaxf(fmaf(v.x, u[q], v.y), fl);
                y[2 * k + 1] = fmaxf(fmaf(v.z, u[q], v.w), fl);
            }
            w = make_uint4(pack_bf16x2(y[0], y[1]), pack_bf16x2(y[2], y[3]), pack_bf16x2(y[4], y[5]),
                           pack_bf16x2(y[6], y[7]));
            if (q < PP) {  // with the bf16 phi that the numerator uses
                const __nv_bfloat162 *yb = reinterpret_cast<const __nv_bfloat162 *>(&w);
#pragma unroll
                for (int k = 0; k < 4; ++k) {
                    dot = fmaf(__low2float(yb[k]), sz[8 * i + 2 * k], dot);
                    dot = fmaf(__high2float(yb[k]), sz[8 * i + 2 * k + 1], dot);
                }
            }
        }
        *reinterpret_cast<uint4 *>((q < PP ? tq : tk) + (i / 8) * C::TILE + sw128_chunk(r, i % 8)) = w;
    }
    return dot;
}

// 32 fp32 values -> bf16 into row f of an MN-major operand whose 64-wide column
// blocks are TILE bytes apart (columns c0 .. c0+31).
template <class C>
__device__ __forceinline__ void store_row32(uint8_t *op, int f, int c0, const float (&v)[32]) {
    uint8_t *blk = op + (c0 / 64) * C::TILE;
    const int ch0 = (c0 % 64) / 8;
#pragma unroll
    for (int k = 0; k < 4; ++k)
        *reinterpret_cast<uint4 *>(blk + sw128_chunk(f, ch0 + k)) =
            make_uint4(pack_bf16x2(v[8 * k], v[8 * k + 1]), pack_bf16x2(v[8 * k + 2], v[8 * k + 3]),
                       pack_bf16x2(v[8 * k + 4], v[8 * k + 5]), pack_bf16x2(v[8 * k + 6], v[8 * k + 7]));
}

template <class C>
__global__ void __launch_bounds__(kCThreads, 1)
    k_tc_causal(const __grid_constant__ CUtensorMap mapQ, const __grid_constant__ CUtensorMap mapK,
                const __grid_constant__ CUtensorMap mapV, AttnArgs a, int *status) {
    extern __shared__ uint8_t smem_raw[];
    uint8_t *sm = align1024(smem_raw);
    uint8_t *Xb = sm;                 // Q tile, then K tile
    uint8_t *Vb = Xb + C::XT;
    uint8_t *Pq = Vb + C::VT;         // phi(Q), then the masked scores A (bf16)
    uint8_t *Pk = Pq + C::PT;         // phi(K)
    uint8_t *Sop = Pk + C::PT;        // S (bf16), MN-major
    uint8_t *Ones = Sop + C::ST;
    uint8_t *Wop = Ones + C::ONES;
    float *sTe = reinterpret_cast<float *>(Wop + C::WOP);
    float *sAB = sTe + kEytzinger;
    float *sbias = sAB + kNint * 16;
    float *sz = sbias + 32;           // z before the current tile
    float *zpre = sz + C::D;          // z at the start of the current segment
    float *sred = zpre + C::D;        // [4 parts][128 rows] normaliser parts
    uint64_t *bars = reinterpret_cast<uint64_t *>(sred + 4 * 128);
    uint64_t *fullx = bars, *xfree = bars + 1, *fullv = bars + 2, *vfree = bars + 3;
    uint64_t *uready = bars + 4, *ufree = bars + 5, *pready = bars + 6, *sready = bars + 7;
    uint64_t *aready = bars + 8, *a2ready = bars + 9, *oready = bars + 10;
    uint32_t *tslot = reinterpret_cast<uint32_t *>(bars + 11);

    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;

    if (tid == 0) {
        mbar_init(fullx, 1); mbar_init(xfree, 1); mbar_init(fullv, 1); mbar_init(vfree, 1);
        mbar_init(uready, 1); mbar_init(ufree, kCWorkers); mbar_init(pready, kCWorkers);
        mbar_init(sready, kCWorkers); mbar_init(aready, 1); mbar_init(a2ready, kCWorkers); mbar_init(oready, 1);
        fence_mbar_init();
    }
    if (warp == 0) { tmem_alloc(tslot, 512); tmem_relinquish(); }
    stage_phi_table<C>(a, sTe, sAB, sbias, Wop);
    for (int e = tid; e < (int)(C::ONES / 4); e += blockDim.x)
        reinterpret_cast<uint32_t *>(Ones)[e] = 0x3F803F80u;  // bf16 1.0 pairs
    grid_dependency_sync();  // the segment prefixes are read, O written from here on
    const Items it(a);
    // padded rows of every item get O = 0
    for (int item = it.begin; item < it.end; ++item) {
        const ItemRange ir = item_range(a, it, item);
        __nv_bfloat16 *O = static_cast<__nv_bfloat16 *>(a.O) + head_rows(a, ir.bh) * C::DV;
        const int z0 = max(ir.r0, ir.r1);
        for (int e = tid; e < (ir.rend - z0) * C::DV / 8; e += blockDim.x)
            reinterpret_cast<uint4 *>(O + (size_t)z0 * C::DV)[e] = make_uint4(0, 0, 0, 0);
    }
    fence_proxy_async_smem();
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tbase = *tslot;
    const int T = block_tiles(a, it);

    if (warp == kCTma) {
        if (lane < 2) {
            TileCursor cur;
            cur.start(a, it);
            bool failed = false;
            for (int g = 0; g < T && !failed; ++g, cur.next(a, it)) {
                if (lane == 0) {
                    // X buffer: load 2g = Q(g), load 2g+1 = K(g); each waits for the projection of the previous load
                    for (int h = 0; h < 2 && !failed; ++h) {
                        const int L = 2 * g + h;
                        if (L >= 1) wait_or_fail(xfree, (L - 1) & 1, failed, status);
                        mbar_arrive_expect_tx(fullx, C::XT);
                        for (int kb = 0; kb < C::KBX; ++kb)
                            tma_load_3d(Xb + kb * C::TILE, h == 0 ? &mapQ : &mapK, kb * 64, cur.row0(), cur.g.bh, fullx);
                    }
                } else {
                    if (g >= 1) wait_or_fail(vfree, (g - 1) & 1, failed, status);
                    mbar_arrive_expect_tx(fullv, C::VT);
                    for (int vb = 0; vb < 2; ++vb)
                        tma_load_3d(Vb + vb * C::TILE, &mapV, vb * 64, cur.row0(), cur.g.bh, fullv);
                }
            }
        }
    } else if (warp == kCMma) {
        if (lane == 0) {
            const uint64_t dX = sdesc(smem_u32(Xb), 16, 1024, kSwizzle128);
            const uint64_t dW = sdesc(smem_u32(Wop), 16, 1024, kSwizzle128);
            const uint64_t dPqK = sdesc(smem_u32(Pq), 16, 1024, kSwizzle128);       // K-major (rows = queries)
            const uint64_t dPkK = sdesc(smem_u32(Pk), 16, 1024, kSwizzle128);       // K-major (rows = keys)
            const uint64_t dPkM = sdesc(smem_u32(Pk), C::TILE, 1024, kSwizzle128);  // MN-major (M = features)
            const uint64_t dV = sdesc(smem_u32(Vb), C::TILE, 1024, kSwizzle128);    // MN-major (N = values)
            const uint64_t dS = sdesc(smem_u32(Sop), C::TILE, 1024, kSwizzle128);   // MN-major (N = values)
            const uint64_t dO1 = sdesc(smem_u32(Ones), 16, 1024, kSwizzle128);      // K-major, 16 rows
            bool failed = false;
            // projections of tile g: U_q from load 2g (into the q slot of g's parity), U_k from load 2g+1
            auto proj = [&](int g, int h) {
                constexpr uint32_t idU = idesc_bf16(128, C::NU, false, false);
                const int L = 2 * g + h;
                wait_or_fail(fullx, L & 1, failed, status);
                tc_fence_after();
                const uint32_t col = h == 0 ? col_uq(g) : cU + C::NU;
#pragma unroll
                for (int kb = 0; kb < C::KBX; ++kb)
#pragma unroll
                    for (int k = 0; k < 4; ++k)
                        mma_bf16_ss(tbase + col, dadd(dX, kb * C::TILE + 32 * k), dadd(dW, kb * (C::NU * 128) + 32 * k),
                                    idU, (kb | k) != 0);
                mma_commit(xfree);
                if (h == 1) mma_commit(uready);
            };
            if (T > 0) { proj(0, 0); proj(0, 1); }
            TileCursor cur;
            cur.start(a, it);
            int tile_in_item = 0, last_item = -1;
            for (int g = 0; g < T && !failed; ++g, cur.next(a, it)) {
                if (cur.item != last_item) { last_item = cur.item; tile_in_item = 0; }
                wait_or_fail(pready, g & 1, failed, status);
                wait_or_fail(sready, g & 1, failed, status);
                tc_fence_after();
                // num = phi(Q) S ;  A = phi(Q) phi(K)^T   (K = 128 features in two 64-blocks)
                constexpr uint32_t idNS = idesc_bf16(128, C::DV, false, true);
                constexpr uint32_t idA = idesc_bf16(128, 128, false, false);
#pragma unroll
                for (int kk = 0; kk < 8; ++kk) {
                    const uint32_t ka = (kk / 4) * C::TILE + 32 * (kk % 4);
                    mma_bf16_ss(tbase + cN, dadd(dPqK, ka), dadd(dS, 2048 * kk), idNS, kk != 0);
                }
#pragma unroll
                for (int kk = 0; kk < 8; ++kk) {
                    const uint32_t ka = (kk / 4) * C::TILE + 32 * (kk % 4);
                    mma_bf16_ss(tbase + cA, dadd(dPqK, ka), dadd(dPkK, ka), idA, kk != 0);
                }
                mma_commit(aready);
                // U_q of the next tile into the other q slot (its Q tile was loaded once U_k(g) freed the X
                // buffer), so that the load of its K tile starts now
                if (g + 1 < T) proj(g + 1, 0);
                wait_or_fail(a2ready, g & 1, failed, status);
                wait_or_fail(fullv, g & 1, failed, status);
                tc_fence_after();
                // num += A V ; S += phi(K)^T V ; z += phi(K)^T 1   (K = 128 keys)
                constexpr uint32_t idAV = idesc_bf16(128, C::DV, false, true);
                constexpr uint32_t idSV = idesc_bf16(128, C::DV, true, true);
                constexpr uint32_t idZ = idesc_bf16(128, 16, true, false);
#pragma unroll
                for (int kk = 0; kk < 8; ++kk) {
                    const uint32_t ka = (kk / 4) * C::TILE + 32 * (kk % 4);
                    mma_bf16_ss(tbase + cN, dadd(dPqK, ka), dadd(dV, 2048 * kk), idAV, 1u);
                }
#pragma unroll
                for (int kk = 0; kk < 8; ++kk) mma_bf16_ss(tbase + cS, dadd(dPkM, 2048 * kk), dadd(dV, 2048 * kk), idSV, 1u);
#pragma unroll
                for (int kk = 0; kk < 8; ++kk)
                    mma_bf16_ss(tbase + cZ, dadd(dPkM, 2048 * kk), dadd(dO1, (kk / 4) * 2048 + 32 * (kk % 4)), idZ,
                                (tile_in_item > 0 || kk > 0) ? 1u : 0u);
                mma_commit(oready);
                mma_commit(vfree);
                // U_k of the next tile (the workers have read U_k(g): they arrived on ufree in phase 1), while
                // they write O and the state operand
                if (g + 1 < T) {
                    wait_or_fail(ufree, g & 1, failed, status);
                    proj(g + 1, 1);
                }
                ++tile_in_item;
            }
        }
    } else {
        // workers: thread (Qd, r) owns row r of the tile and feature / column quarter Qd
        const int Qd = warp >> 2, r = ((warp & 3) << 5) | lane;
        const uint32_t lrow = (uint32_t)((warp & 3) << 5) << 16;
        bool failed = false;
        int g = 0;
        for (int item = it.begin; item < it.end; ++item) {
            const ItemRange ir = item_range(a, it, item);
            if (ir.ntiles == 0) continue;
            // segment start: S (TMEM, fp32) and its bf16 operand from the prefix state, z from the prefix sums
            {
                const float *Sp = a.seg_S + (head_state(a, ir.bh) * (a.nseg + 1) + ir.chunk) * C::D * C::DV;
                const int f = r, c0 = 32 * Qd;  // TMEM lane f (feature), columns c0 .. c0+31
                float v[32];
#pragma unroll
                for (int c = 0; c < 32; c += 4) {
                    const float4 x = __ldcg(reinterpret_cast<const float4 *>(Sp + (size_t)f * C::DV + c0 + c));
                    v[c] = x.x; v[c + 1] = x.y; v[c + 2] = x.z; v[c + 3] = x.w;
                }
                uint32_t w0[16], w1[16];
#pragma unroll
                for (int c = 0; c < 16; ++c) { w0[c] = __float_as_uint(v[c]); w1[c] = __float_as_uint(v[16 + c]); }
                tmem_st16(tbase + lrow + cS + c0, w0);
                tmem_st16(tbase + lrow + cS + c0 + 16, w1);
                tmem_wait_st();
                store_row32<C>(Sop, f, c0, v);
                if (Qd == 0) {
                    const float zv = __ldcg(a.seg_z + (head_state(a, ir.bh) * (a.nseg + 1) + ir.chunk) * C::D + f);
                    zpre[f] = zv;
                    sz[f] = zv;
                }
                fence_proxy_async_smem();
                tc_fence_before();
                mbar_arrive(sready);
                named_sync<kCWorkers>(1);  // sz of the segment start
            }
            __nv_bfloat16 *O = static_cast<__nv_bfloat16 *>(a.O) + head_rows(a, ir.bh) * C::DV;
            for (int t = 0; t < ir.ntiles; ++t, ++g) {
                const int row0 = ir.r0 + t * 128;
                const int nvalid = min(128, ir.r1 - row0);
                const bool valid = r < nvalid;
                const bool last = t == ir.ntiles - 1;
                // phase 1: phi(Q), phi(K), phi(q).z
                wait_or_fail(uready, g & 1, failed, status);
                tc_fence_after();
                const float dq = phi_quarter_qk<C>(tbase + lrow + col_uq(g), tbase + lrow + cU + C::NU, Qd, sTe, sAB,
                                                   sbias, channel_floor(a.lay), valid, r, Pq, Pk, sz);
                tc_fence_before();
                mbar_arrive(ufree);
                if (!valid && Qd == 0) {  // padded key rows: clear V so that no garbage enters num or S
                    wait_or_fail(fullv, g & 1, failed, status);
#pragma unroll
                    for (int vb = 0; vb < 2; ++vb)
#pragma unroll
                        for (int c = 0; c < 8; ++c)
                            *reinterpret_cast<uint4 *>(Vb + vb * C::TILE + sw128_chunk(r, c)) = make_uint4(0, 0, 0, 0);
                }
                fence_proxy_async_smem();
                tc_fence_before();
                mbar_arrive(pready);
                // phase 2: A masked to keys j <= r, row sums, bf16 into the phi(Q) tile
                wait_or_fail(aready, g & 1, failed, status);
                tc_fence_after();
                float den = dq;
                {
                    const int j0 = 32 * Qd;
                    uint32_t x0[16], x1[16];
                    tmem_ld16(tbase + lrow + cA + j0, x0);
                    tmem_ld16(tbase + lrow + cA + j0 + 16, x1);
                    tmem_wait_ld();
                    float v[32];  // rounded to bf16 as the numerator's A V uses them
#pragma unroll
                    for (int c = 0; c < 16; ++c) {
                        v[c] = (valid && j0 + c <= r) ? __bfloat162float(__float2bfloat16_rn(__uint_as_float(x0[c]))) : 0.0f;
                        v[16 + c] =
                            (valid && j0 + 16 + c <= r) ? __bfloat162float(__float2bfloat16_rn(__uint_as_float(x1[c]))) : 0.0f;
                    }
#pragma unroll
                    for (int c = 0; c < 32; ++c) den += v[c];
                    store_row32<C>(Pq, r, j0, v);  // K-major A: row r, key columns j0 ..
                }
                sred[Qd * 128 + r] = den;
                fence_proxy_async_smem();
                tc_fence_before();
                mbar_arrive(a2ready);
                // phase 3: O, then the state operand of the next tile
                wait_or_fail(oready, g & 1, failed, status);
                tc_fence_after();
                named_sync<kCWorkers>(1);  // normaliser parts
                const float dsum = ((sred[r] + sred[128 + r]) + (sred[256 + r] + sred[384 + r])) + a.eps;
                {
                    uint32_t x0[16], x1[16];
                    tmem_ld16(tbase + lrow + cN + 32 * Qd, x0);
                    tmem_ld16(tbase + lrow + cN + 32 * Qd + 16, x1);
                    tmem_wait_ld();
                    if (valid) {
                        const float inv = dsum != 0.0f ? 1.0f / dsum : 0.0f;  // one division per row
                        float o[32];
#pragma unroll
                        for (int c = 0; c < 16; ++c) {
                            o[c] = __uint_as_float(x0[c]) * inv;
                            o[16 + c] = __uint_as_float(x1[c]) * inv;
                        }
                        uint4 *dst = reinterpret_cast<uint4 *>(O + (size_t)(row0 + r) * C::DV + 32 * Qd);
#pragma unroll
                        for (int k = 0; k < 4; ++k)
                            dst[k] = make_uint4(pack_bf16x2(o[8 * k], o[8 * k + 1]), pack_bf16x2(o[8 * k + 2], o[8 * k + 3]),
                                                pack_bf16x2(o[8 * k + 4], o[8 * k + 5]),
                                                pack_bf16x2(o[8 * k + 6], o[8 * k + 7]));
                    }
                }
                if (!last) {
                    // S after this tile -> bf16 operand; z -> sz
                    const int f = r, c0 = 32 * Qd;
                    uint32_t x0[16], x1[16];
                    tmem_ld16(tbase + lrow + cS + c0, x0);
                    tmem_ld16(tbase + lrow + cS + c0 + 16, x1);
                    tmem_wait_ld();
                    float v[32];
#pragma unroll
                    for (int c = 0; c < 16; ++c) { v[c] = __uint_as_float(x0[c]); v[16 + c] = __uint_as_float(x1[c]); }
                    store_row32<C>(Sop, f, c0, v);
                    if (Qd == 0) {
                        uint32_t zx[4];
                        tmem_ld4(tbase + lrow + cZ, zx);
                        tmem_wait_ld();
                        sz[f] = zpre[f] + __uint_as_float(zx[0]);
                    }
                    fence_proxy_async_smem();
                    tc_fence_before();
                    mbar_arrive(sready);
                }
                named_sync<kCWorkers>(1);  // sz, and sred free for the next tile
            }
        }
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 0) tmem_dealloc(tbase, 512);
}

// Exclusive prefix of the segment statistics at every segment start, total last:
// seg_S[bh][s] = sum_{s' < s} S_part[bh][s'] (s = 0 .. nseg), in segment order.
__global__ void __launch_bounds__(256) k_seg_scan(AttnArgs a) {
    grid_dependency_sync();
    const int bh = blockIdx.y;
    const size_t SD = (size_t)a.D * a.dv;
    const int e4 = blockIdx.x * blockDim.x + threadIdx.x;  // float4 position
    if ((size_t)e4 * 4 < SD) {
        const float4 *part = reinterpret_cast<const float4 *>(a.S_part + (size_t)bh * a.nseg * SD) + e4;
        float4 *out = reinterpret_cast<float4 *>(a.seg_S + head_state(a, bh) * (a.nseg + 1) * SD) + e4;
        float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
        for (int s = 0; s < a.nseg; ++s) {
            const float4 v = __ldcg(part + (size_t)s * (SD / 4));
            out[(size_t)s * (SD / 4)] = acc;
            acc.x += v.x; acc.y += v.y; acc.z += v.z; acc.w += v.w;
        }
        out[(size_t)a.nseg * (SD / 4)] = acc;
    }
    if (blockIdx.x == 0) {
        for (int f = threadIdx.x; f < a.D; f += blockDim.x) {
            const float *part = a.z_part + (size_t)bh * a.nseg * a.D + f;
            float *out = a.seg_z + head_state(a, bh) * (a.nseg + 1) * a.D + f;
            float acc = 0.0f;
            for (int s = 0; s < a.nseg; ++s) {
                const float v = __ldcg(part + (size_t)s * a.D);
                out[(size_t)s * a.D] = acc;
                acc += v;
            }
            out[(size_t)a.nseg * a.D] = acc;
        }
    }
}

}  // namespace

bool tc_make_map(CUtensorMap *m, const void *base, int width, int n, int BH, int hs_mul);
int tc_sm_count();

bool tc_causal_supported(const luna_attn_desc &ad, const TableLayout &lay) {
    return ad.io == LUNA_BF16 && ad.causal && lay.L == 8 && lay.P <= 512 && ad.d == 128 && ad.dv == 128 && lay.M == 16;
}

cudaError_t launch_tc_causal_stats(const AttnArgs &a0, cudaStream_t s) {
    AttnArgs a = a0;
    a.rows_per_split = a0.seg_len;  // work item = state segment (whole 128-row tiles)
    a.nsplit = a0.nseg;
    cudaError_t e = launch_tc_keys_items(a, s);
    if (e != cudaSuccess) return e;
    const size_t SD4 = (size_t)a.D * a.dv / 4;
    LUNA_LAUNCH_DEP("seg_scan", !a.ch_sigma, k_seg_scan, dim3((unsigned)((SD4 + 255) / 256), a.B * a.H), 256, 0, s, a);
    return cudaGetLastError();
}

cudaError_t launch_tc_causal_fwd(const AttnArgs &a0, cudaStream_t s) {
    using C = K128;
    AttnArgs a = a0;
    a.rows_per_split = a0.seg_len;  // work item = state segment (whole 128-row tiles)
    a.nsplit = a0.nseg;
    cudaError_t e = launch_tc_causal_stats(a, s);
    if (e != cudaSuccess) return e;
    const int BH = a.B * a.H;
    CUtensorMap mQ, mK, mV;
    if (!tc_make_map(&mQ, a.Q, a.d, a.n, BH, a.hs_mul) || !tc_make_map(&mK, a.K, a.d, a.n, BH, a.hs_mul) ||
        !tc_make_map(&mV, a.V, a.dv, a.n, BH, a.hs_mul))
        return cudaErrorInvalidValue;
    if ((e = cudaFuncSetAttribute(k_tc_causal<C>, cudaFuncAttributeMaxDynamicSharedMemorySize, C::SMEM)) != cudaSuccess)
        return e;
    const int items = BH * a.nsplit;
    const int grid = items < tc_sm_count() ? items : tc_sm_count();
    int *st = reinterpret_cast<int *>(reinterpret_cast<char *>(a.counters) - 256);
    LUNA_LAUNCH_DEP("tc_causal", !a.ch_sigma, k_tc_causal<C>, grid, kCThreads, C::SMEM, s, mQ, mK, mV, a, st);
    return cudaGetLastError();
}

}  // namespace luna
