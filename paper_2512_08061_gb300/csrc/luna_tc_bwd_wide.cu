// Tensor-core backward pass for full 128-byte rows: bf16 I/O, non-causal,
// d = dv = 64, M = 8 projections, L = 8 channels (D = 64).
//
// The same computation as the d = 32 kernels (see luna_tc_bwd.cu), with the
// layout that full rows force:
//   - dO fills its tile, so G = [dU_hi | dU_lo | dU_hi | 0 | -(dO.O) hi, lo | 0]
//     gets a tile of its own, and dz comes from a second contraction
//     [phi/den]^T G (G columns 32..47) next to dS = [phi/den]^T dO;
//   - the projection operand uses all 64 columns of its rows, so the dX operand
//     [W_hi; W_hi; W_lo; 0] (64 output columns) has a region of its own;
//   - tensor memory holds one P (query side) and one dphi and one dV (key side):
//     the MMA warp issues the next tile's P or dphi once the workers have
//     released the current one (they read it before handing over G).
// Query side per tile: U = Q [W_hi; W_mid; W_lo]^T, P = dO [S_hi; S_lo]^T;
// workers phi, den, dO.O, dphi, dU, histogram, G; MMA dS += [phi/den]^T dO,
// dz += [phi/den]^T G', dW^T += Q^T dU, dQ = dU W.
// Key side per tile: U = K [...]^T, dphi = V [dS_hi; dS_lo]^T, dV = phi [dS_hi; dS_lo];
// workers dphi + dz, dU, histogram, G; MMA dK = dU W, dW^T += K^T dU.
#include "luna_tc_bwd_dev.cuh"

namespace luna {
namespace {
using namespace sm100;
using namespace simt;
using namespace tcdev;
using namespace tcbwd;

struct B64 {
    static constexpr int d = 64, DX = 64, DV = 64, MP = 8, D = 64, NU = 32, PP = MP / kBRowThreads;
    static constexpr uint32_t TILE = 16384;  // 128 rows x 128 B
    static constexpr int NKD = d / 16;
    static constexpr int NKV = DV / 16;
    static constexpr uint32_t WOP = NU * 128;          // [W_hi; W_mid; W_lo; 0] x 64 input columns
    static constexpr uint32_t WXP = d * 128;           // dX operand, 64 output-column rows (K = 32 used)
    static constexpr uint32_t SOP2 = 2 * D * 128;      // [S_hi; S_lo] rows per feature, K = dv = 64
    static constexpr uint32_t SOP = 2 * DV * 128;      // [S_hi; S_lo]^T rows per value column, K = D = 64
    static constexpr uint32_t HIST = kNint * 16 * 4;
    static constexpr uint32_t SRED = 2 * 2 * kBRowThreads * 128;
    static constexpr uint32_t SMAX = 2 * (kBWorkers / 32) * 4;
    static constexpr uint32_t MISC = D * 4 + MP * d * 4 + 64 + SMAX + kBarBytes + 1024;
    // query: Q tiles x 2, phi/den tiles (hi, lo interleaved by 16 features) x 1, dO tiles x 2, G x 1
    static constexpr int NSQ = 2, NOQ = 2;
    static constexpr uint32_t SMEM_Q = NSQ * TILE + 2 * TILE + NOQ * TILE + TILE + WOP + WXP + SOP2 + kTableBytes +
                                       SRED * 4 + HIST + MISC;
    // key: [phi | K] stages x 2, V x 1, G x 1
    static constexpr int NSK = 2;
    static constexpr uint32_t SMEM_K = NSK * 2 * TILE + TILE + TILE + WOP + WXP + SOP + SOP2 + kTableBytes + HIST + MISC;
    static_assert(SMEM_Q <= kSmemLimit && SMEM_K <= kSmemLimit, "shared memory budget");
};

// ---------------------------------------------------------------------------
// query side

template <class C>
__global__ void __launch_bounds__(kBThreads, 1)
    k_tc_bwd_query_w(const __grid_constant__ CUtensorMap mapQ, const __grid_constant__ CUtensorMap mapdO, AttnArgs a,
                     int *status) {
    extern __shared__ uint8_t smem_raw[];
    const float fl = channel_floor(a.lay);  // lower bound of a channel output
    uint8_t *sm = align1024(smem_raw);
    constexpr int NS = C::NSQ, NO = C::NOQ;
    constexpr uint32_t T16 = C::TILE;
    uint8_t *Qb = sm;                    // [NS] Q tiles
    uint8_t *Pt = Qb + NS * T16;         // phi/den, two 64-feature tiles (hi, lo interleaved by 16 features)
    uint8_t *Ob = Pt + 2 * T16;          // [NO] dO tiles
    uint8_t *Gt = Ob + NO * T16;         // G = [dU_hi | dU_lo | dU_hi | 0 | -(dO.O) hi, lo | 0]
    uint8_t *Wop = Gt + T16;
    uint8_t *Wx = Wop + C::WOP;
    uint8_t *Sop2 = Wx + C::WXP;
    float *sTe = reinterpret_cast<float *>(Sop2 + C::SOP2);
    float *sAB = sTe + kEytzinger;
    float *sbias = sAB + kNint * 16;
    float *sz = sbias + 32;
    float *sred = sz + C::D;
    int *bins = reinterpret_cast<int *>(sred + C::SRED);
    float *sdW = reinterpret_cast<float *>(bins + kNint * 16);  // [M][d]
    float *sdb = sdW + C::MP * C::d;
    float *smax = sdb + 16;
    uint64_t *bars = reinterpret_cast<uint64_t *>(smax + 2 * (kBWorkers / 32));
    uint64_t *fullq = bars;               // [NS]
    uint64_t *qfree = fullq + NS;         // [NS] projection and dW^T consumed the Q tile
    uint64_t *fullo = qfree + NS;         // [NO]
    uint64_t *ofree = fullo + NO;         // [NO]
    uint64_t *uready = ofree + NO;        // [2]
    uint64_t *pready = uready + 2;        // [1]
    uint64_t *gready = pready + 1;        // [1] count 512
    uint64_t *dqready = gready + 1;       // [1]
    uint64_t *dqfree = dqready + 1;       // [1] count 512
    uint64_t *accdone = dqfree + 1;       // [2]
    uint64_t *accfree = accdone + 2;      // [2] count 128
    uint64_t *opready = accfree + 2;      // [1] count 512
    uint64_t *wdone = opready + 1;        // [1]
    uint32_t *tslot = reinterpret_cast<uint32_t *>(wdone + 1);
    int *slast = reinterpret_cast<int *>(tslot + 1);
    static_assert((2 * NS + 2 * NO + 13) * 8 + 8 <= kBarBytes, "barrier area");

    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const Items it(a);
    // TMEM: U [2 x 32] | P [128] | dS [2 x 64] | dz [2 x 16] | dQ [64] | dW^T (M = 64) [16]
    constexpr uint32_t cU = 0, cP = 64, cA = 192, cZ = 320, cQ = 352, cW = 416;

    if (tid == 0) {
        for (int i = 0; i < NS; ++i) { mbar_init(fullq + i, 1); mbar_init(qfree + i, 1); }
        for (int i = 0; i < NO; ++i) { mbar_init(fullo + i, 1); mbar_init(ofree + i, 1); }
        for (int i = 0; i < 2; ++i) {
            mbar_init(uready + i, 1); mbar_init(accdone + i, 1); mbar_init(accfree + i, 128);
        }
        mbar_init(pready, 1); mbar_init(gready, kBWorkers);
        mbar_init(dqready, 1); mbar_init(dqfree, kBWorkers);
        mbar_init(opready, kBWorkers); mbar_init(wdone, 1);
        fence_mbar_init();
    }
    if (warp == 0) { tmem_alloc(tslot, 512); tmem_relinquish(); }
    stage_phi_table<C>(a, sTe, sAB, sbias, Wop);
    stage_wx<C>(a, Wx, 0);
    for (int e = tid; e < kNint * 16; e += blockDim.x) bins[e] = 0;
    for (int e = tid; e < C::MP * C::d + 16; e += blockDim.x) sdW[e] = 0.0f;
    for (int e = tid; e < (int)(T16 / 16); e += blockDim.x) reinterpret_cast<uint4 *>(Gt)[e] = make_uint4(0, 0, 0, 0);
    float *hpart = a.gpart + (size_t)blockIdx.x * a.gsize + C::MP * a.d + C::MP;
    for (int e = tid; e < a.lay.nint * 16; e += blockDim.x) hpart[e] = 0.0f;
    for (int item = it.begin; item < it.end && !a.padded_zeroed; ++item) {  // padded rows: zero gradients
        const ItemRange ir = item_range(a, it, item);
        __nv_bfloat16 *dQ = static_cast<__nv_bfloat16 *>(a.dQ) + head_rows(a, ir.bh) * C::d;
        const int z0 = max(ir.r0, ir.r1);
        for (int e = tid; e < (ir.rend - z0) * C::d / 8; e += blockDim.x)
            reinterpret_cast<uint4 *>(dQ + (size_t)z0 * C::d)[e] = make_uint4(0, 0, 0, 0);
    }
    fence_proxy_async_smem();
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tbase = *tslot;

    if (warp == kBTma) {
        if (lane < 2) {
            const int T = block_tiles(a, it);
            TileCursor cur;
            cur.start(a, it);
            bool failed = false;
            for (int g = 0; g < T && !failed; ++g, cur.next(a, it)) {
                if (lane == 0) {
                    const int s = g % NS;
                    if (g >= NS) wait_or_fail(qfree + s, ((g - NS) / NS) & 1, failed, status);
                    mbar_arrive_expect_tx(fullq + s, T16);
                    tma_load_3d(Qb + s * T16, &mapQ, 0, cur.row0(), cur.g.bh, fullq + s);
                } else {
                    const int o = g % NO;
                    if (g >= NO) wait_or_fail(ofree + o, ((g - NO) / NO) & 1, failed, status);
                    mbar_arrive_expect_tx(fullo + o, T16);
                    tma_load_3d(Ob + o * T16, &mapdO, 0, cur.row0(), cur.g.bh, fullo + o);
                }
            }
        }
    } else if (warp == kBMma) {
        if (lane == 0) {
            const int T = block_tiles(a, it);
            const uint64_t dQt = sdesc(smem_u32(Qb), 16384, 1024, kSwizzle128);
            const uint64_t dP = sdesc(smem_u32(Pt), 16384, 1024, kSwizzle128);
            const uint64_t dO0 = sdesc(smem_u32(Ob), 16384, 1024, kSwizzle128);
            const uint64_t dG = sdesc(smem_u32(Gt), 16384, 1024, kSwizzle128);
            const uint64_t dWo = sdesc(smem_u32(Wop), 16, 1024, kSwizzle128);
            const uint64_t dWx = sdesc(smem_u32(Wx), 16, 1024, kSwizzle128);
            const uint64_t dSp = sdesc(smem_u32(Sop2), 16, 1024, kSwizzle128);
            bool failed = false;
            auto proj = [&](int g) {
                const int s = g % NS;
                wait_or_fail(fullq + s, (g / NS) & 1, failed, status);
                tc_fence_after();
                proj_mma<C>(tbase + cU + (g & 1) * C::NU, dadd(dQt, s * T16), dWo);
                mma_commit(uready + (g & 1));
            };
            auto pmma = [&](int g) {  // P = dO [S_hi; S_lo]^T into the single P columns
                const int o = g % NO;
                wait_or_fail(fullo + o, (g / NO) & 1, failed, status);
                tc_fence_after();
                constexpr uint32_t idP = idesc_bf16(128, 2 * C::D, false, false);
#pragma unroll
                for (int k = 0; k < C::NKV; ++k)
                    mma_bf16_ss(tbase + cP, dadd(dO0, o * T16 + 32 * k), dadd(dSp, 32 * k), idP, k != 0);
                mma_commit(pready);
            };
            int op_phase = 0;
            if (T > 0) { proj(0); wait_or_fail(opready, op_phase++ & 1, failed, status); pmma(0); }
            if (T > 1) proj(1);
            TileCursor cur;
            cur.start(a, it);
            int run_bh = -1, ne = 0, run_left = 0, tile_in_run = 0;
            for (int g = 0; g < T && !failed; ++g) {
                const int s = g % NS, o = g % NO;
                if (cur.g.bh != run_bh) {
                    run_bh = cur.g.bh;
                    run_left = 0;
                    for (int i = cur.item; i < it.end && i / it.nchunk == run_bh; ++i)
                        run_left += item_range(a, it, i).ntiles;
                    tile_in_run = 0;
                    if (ne >= 2) wait_or_fail(accfree + (ne & 1), ((ne - 2) >> 1) & 1, failed, status);
                }
                const int b = ne & 1;
                TileCursor nx = cur;
                nx.next(a, it);
                const bool next_new_run = (g + 1 < T) && nx.g.bh != cur.g.bh;
                wait_or_fail(gready, g & 1, failed, status);
                if (g >= 1) wait_or_fail(dqfree, (g - 1) & 1, failed, status);
                tc_fence_after();
                // dQ = [dU_hi | dU_lo | dU_hi | 0] W first, its barrier committed at once
                constexpr uint32_t idQ = idesc_bf16(128, C::d, false, false);
#pragma unroll
                for (int k = 0; k < 2; ++k) mma_bf16_ss(tbase + cQ, dadd(dG, 32 * k), dadd(dWx, 32 * k), idQ, k != 0);
                mma_commit(dqready);
                const uint32_t acc = (tile_in_run > 0) ? 1u : 0u;
                // dS += [phi/den hi, lo]^T dO ;  dz += [phi/den hi, lo]^T G (columns 32..47)
                constexpr uint32_t idS = idesc_bf16(128, C::DV, true, true);
                constexpr uint32_t idZ = idesc_bf16(128, 16, true, true);
#pragma unroll
                for (int k = 0; k < 8; ++k) {
                    mma_bf16_ss(tbase + cA + b * C::DV, dadd(dP, 2048 * k), dadd(dO0, o * T16 + 2048 * k), idS,
                                (acc | (k > 0)) ? 1u : 0u);
                    mma_bf16_ss(tbase + cZ + b * 16, dadd(dP, 2048 * k), dadd(dG, 64 + 2048 * k), idZ,
                                (acc | (k > 0)) ? 1u : 0u);
                }
                // dW^T += Q^T [dU_hi | dU_lo] (G columns 0..15)
                constexpr uint32_t idW = idesc_bf16(64, 16, true, true);
#pragma unroll
                for (int k = 0; k < 8; ++k)
                    mma_bf16_ss(tbase + cW, dadd(dQt, s * T16 + 2048 * k), dadd(dG, 2048 * k), idW,
                                (g > 0 || k > 0) ? 1u : 0u);
                mma_commit(ofree + o);
                mma_commit(qfree + s);
                ++tile_in_run;
                if (--run_left == 0) { mma_commit(accdone + b); ++ne; }
                // the workers have read P(g) (before gready): P of the next tile
                if (g + 1 < T) {
                    if (next_new_run) wait_or_fail(opready, op_phase++ & 1, failed, status);
                    pmma(g + 1);
                }
                if (g + 2 < T) proj(g + 2);
                cur = nx;
            }
            if (T > 0 && !failed) mma_commit(wdone);
            else mbar_arrive(wdone);
        }
    } else {
        const int H = warp >> 2, r = ((warp & 3) << 5) | lane;
        const uint32_t lrow = (uint32_t)((warp & 3) << 5) << 16;
        bool failed = false;
        float db_acc[C::PP];
#pragma unroll
        for (int q = 0; q < C::PP; ++q) db_acc[q] = 0.0f;
        HistAcc hacc;
        // dQ of tile g is read out during tile g + 1 (after its feature-map work, before its G tile), so
        // that the dQ product runs while the workers start the next tile
        int pend_g = -1, pend_row = -1;  // tile, and this thread's row of [B*H*n] in it (-1: padded; the
                                         // rows of tensors that fit in device memory stay below 2^31)
        auto dq_out = [&](int gp, int row) {
            wait_or_fail(dqready, gp & 1, failed, status);
            tc_fence_after();
            uint32_t x[16];
            tmem_ld16(tbase + lrow + cQ + H * 16, x);
            tmem_wait_ld();
            float f0[8], f1[8];
#pragma unroll
            for (int c = 0; c < 8; ++c) { f0[c] = __uint_as_float(x[c]); f1[c] = __uint_as_float(x[8 + c]); }
            tc_fence_before();
            mbar_arrive(dqfree);
            if (row >= 0) {
                uint4 *dst = reinterpret_cast<uint4 *>(static_cast<__nv_bfloat16 *>(a.dQ) + (size_t)row * C::d + H * 16);
                dst[0] = pack8(f0);
                dst[1] = pack8(f1);
            }
        };
        int g = 0, ne = 0;
        for (int i0 = it.begin; i0 < it.end;) {
            const int bh = i0 / it.nchunk;
            const int i1 = min(it.end, (bh + 1) * it.nchunk);
            int run_tiles = 0;
            for (int i = i0; i < i1; ++i) run_tiles += item_range(a, it, i).ntiles;
            if (run_tiles > 0) {  // operands of this head: [S_hi; S_lo] rows per feature, z
                named_sync<kBWorkers>(1);
                stage_rows_per_feature<C>(a.S_fin + head_state(a, bh) * C::D * C::DV, Sop2, tid, kBWorkers);
                for (int e = tid; e < C::D; e += kBWorkers) sz[e] = a.z_fin[head_state(a, bh) * C::D + e];
                fence_proxy_async_smem();
                named_sync<kBWorkers>(1);
                mbar_arrive(opready);
            }
            for (int item = i0; item < i1; ++item) {
                const ItemRange ir = item_range(a, it, item);
                for (int t = 0; t < ir.ntiles; ++t, ++g) {
                    const int s = g % NS, o = g % NO;
                    const int row0 = ir.r0 + t * 128;
                    const int nvalid = min(128, ir.r1 - row0);
                    const bool valid = r < nvalid;
                    uint8_t *qt = Qb + s * T16, *ot = Ob + o * T16;
                    wait_or_fail(uready + (g & 1), (g >> 1) & 1, failed, status);
                    tc_fence_after();
                    float u[C::PP];
                    int j[C::PP];
                    {
                        static_assert(C::PP == 2, "two projections per thread");
                        uint32_t xh[2], xm[2], xl[2];
                        const uint32_t ucol = tbase + lrow + cU + (g & 1) * C::NU + H * C::PP;
                        tmem_ld2(ucol, xh);
                        tmem_ld2(ucol + C::MP, xm);
                        tmem_ld2(ucol + 2 * C::MP, xl);
                        tmem_wait_ld();
#pragma unroll
                        for (int q = 0; q < C::PP; ++q)
                            u[q] = (__uint_as_float(xh[q]) + __uint_as_float(xm[q])) + __uint_as_float(xl[q]) +
                                   sbias[H * C::PP + q];
                    }
                    search<C::PP>(sTe, u, j);
                    if (!valid && H == 0) zero_row(qt, r);  // padded rows: no contribution to dW
                    // normaliser and dO.O from P = S dO
                    wait_or_fail(pready, g & 1, failed, status);
                    tc_fence_after();
                    float denp = 0.0f, dotp = 0.0f;
#pragma unroll
                    for (int q = 0; q < C::PP; ++q) {
                        const int i = H * C::PP + q;
                        float al[8], y[8];
                        channel_eval(sAB, j[q], u[q], fl, al, y);
                        uint32_t ph[8], pl[8];
                        tmem_ld8(tbase + lrow + cP + 8 * i, ph);
                        tmem_ld8(tbase + lrow + cP + C::D + 8 * i, pl);
                        tmem_wait_ld();
#pragma unroll
                        for (int l = 0; l < 8; ++l) {
                            denp = fmaf(y[l], sz[8 * i + l], denp);
                            dotp = fmaf(y[l], __uint_as_float(ph[l]) + __uint_as_float(pl[l]), dotp);
                        }
                    }
                    float *rs = sred + (g & 1) * (C::SRED / 2);
                    rs[H * 128 + r] = denp;
                    rs[kBRowThreads * 128 + H * 128 + r] = dotp;
                    quarter_sync(warp);  // the parts of this quarter's rows
                    float den = a.eps, dotn = 0.0f;
#pragma unroll
                    for (int h = 0; h < kBRowThreads; ++h) {
                        den += rs[h * 128 + r];
                        dotn += rs[kBRowThreads * 128 + h * 128 + r];
                    }
                    const bool live = valid && den != 0.0f;
                    const float inv = live ? 1.0f / den : 0.0f;
                    const float ndot = live ? -dotn * inv : 0.0f;  // -(dO.O)
                    const float dden = ndot * inv;
                    bool hon = hacc.open;
                    // gradients through the feature map; phi/den (bf16 hi, lo) for the dS / dz contractions
                    float dU[C::PP], gv[C::PP][8];
#pragma unroll
                    for (int q = 0; q < C::PP; ++q) {
                        const int i = H * C::PP + q;
                        float al[8], y[8];
                        channel_eval(sAB, j[q], u[q], fl, al, y);
                        {
                            float yh[8], yl[8];
#pragma unroll
                            for (int l = 0; l < 8; ++l) {
                                const float v = live ? y[l] * inv : 0.0f;
                                yh[l] = __bfloat162float(__float2bfloat16_rn(v));
                                yl[l] = v - yh[l];
                            }
                            const int ch = 4 * (i >> 1) + (i & 1), cl = ch + 2;
                            *reinterpret_cast<uint4 *>(Pt + (ch >> 3) * T16 + sw128_chunk(r, ch & 7)) = pack8(yh);
                            *reinterpret_cast<uint4 *>(Pt + (cl >> 3) * T16 + sw128_chunk(r, cl & 7)) = pack8(yl);
                        }
                        uint32_t ph[8], pl[8];
                        tmem_ld8(tbase + lrow + cP + 8 * i, ph);
                        tmem_ld8(tbase + lrow + cP + C::D + 8 * i, pl);
                        tmem_wait_ld();
                        float du = 0.0f;
#pragma unroll
                        for (int l = 0; l < 8; ++l) {
                            const float dphi =
                                live ? (__uint_as_float(ph[l]) + __uint_as_float(pl[l])) * inv + sz[8 * i + l] * dden : 0.0f;
                            const float gl = y[l] > fl ? dphi : 0.0f;
                            gv[q][l] = gl;
                            du = fmaf(gl, al[l], du);
                        }
                        dU[q] = du;
                        db_acc[q] += du;
                    }
                    if (pend_g >= 0) dq_out(pend_g, pend_row);
                    // G and the dO rows of padded rows (which the dS contraction reads)
                    {
                        if (!valid) {
#pragma unroll
                            for (int c = 0; c < 2; ++c)
                                *reinterpret_cast<uint4 *>(ot + sw128_chunk(r, 2 * H + c)) = make_uint4(0, 0, 0, 0);
                        }
                        uint32_t vh, vl;
                        dU_pack(dU, vh, vl);
                        *reinterpret_cast<uint32_t *>(Gt + sw128_chunk(r, 0) + H * 4) = vh;
                        *reinterpret_cast<uint32_t *>(Gt + sw128_chunk(r, 1) + H * 4) = vl;
                        *reinterpret_cast<uint32_t *>(Gt + sw128_chunk(r, 2) + H * 4) = vh;
                        if (H == 0) {  // chunk 4: -(dO.O) as hi, lo (chunks 3, 5 stay zero)
                            __nv_bfloat16 th, tl;
                            split_bf16(ndot, th, tl);
                            *reinterpret_cast<uint4 *>(Gt + sw128_chunk(r, 4)) = make_uint4(
                                (uint32_t)__bfloat16_as_ushort(th) | ((uint32_t)__bfloat16_as_ushort(tl) << 16), 0u, 0u, 0u);
                        }
                    }
                    fence_proxy_async_smem();
                    tc_fence_before();
                    mbar_arrive(gready);
                    if (!hon) {  // first tile with a nonzero g in the block: its maxima give the first scales
                        float m0 = 0.0f, m1 = 0.0f;
#pragma unroll
                        for (int q = 0; q < C::PP; ++q)
#pragma unroll
                            for (int l = 0; l < 8; ++l) {
                                m0 = finite_max(m0, gv[q][l]);
                                m1 = finite_max(m1, gv[q][l] * u[q]);
                            }
                        hon = hist_open(hacc, m0, m1, smax, warp, lane);
                    }
                    if (hon) {
                        hist_add<C::PP>(bins, hpart, hacc, j, u, gv, dU);
                        if (++hacc.tiles == hist_tiles<C::MP>()) hist_close(bins, hpart, a.lay.nint, hacc, tid, true, smax, warp, lane);
                    }
                    pend_g = g;
                    pend_row = valid ? (int)head_rows(a, bh) + row0 + r : -1;
                }
            }
            // run epilogue (warps 0..3): dS, dz partial of this head; warp w holds features 16w..16w+15,
            // hi in lanes 0..15 and lo in lanes 16..31
            if (warp < 4) {
                const RunSlot rs = run_slot(a, it, bh);
                const int nruns = rs.nruns;
                const size_t slot = (size_t)bh * it.nchunk + rs.rank;
                float *Sp = a.dS_part + slot * C::D * C::DV;
                float *zp = a.dz_part + slot * C::D;
                const uint32_t lr = (uint32_t)(warp << 5) << 16;
                const bool have = run_tiles > 0;
                const int b = ne & 1;
                if (have) wait_or_fail(accdone + b, (ne >> 1) & 1, failed, status);
                tc_fence_after();
                const int f = (warp << 4) | (lane & 15);
#pragma unroll
                for (int c0 = 0; c0 < C::DV; c0 += 16) {
                    uint32_t x[16];
                    if (have) { tmem_ld16(tbase + lr + cA + b * C::DV + c0, x); tmem_wait_ld(); }
                    float fx[16];
#pragma unroll
                    for (int c = 0; c < 16; ++c) {
                        fx[c] = have ? __uint_as_float(x[c]) : 0.0f;
                        fx[c] += __shfl_down_sync(0xffffffffu, fx[c], 16);
                    }
                    if (lane < 16) {
#pragma unroll
                        for (int c = 0; c < 16; c += 4)
                            *reinterpret_cast<float4 *>(Sp + f * C::DV + c0 + c) =
                                make_float4(fx[c], fx[c + 1], fx[c + 2], fx[c + 3]);
                    }
                }
                {
                    uint32_t zx[4];
                    if (have) { tmem_ld4(tbase + lr + cZ + b * 16, zx); tmem_wait_ld(); }
                    float fz = have ? __uint_as_float(zx[0]) + __uint_as_float(zx[1]) : 0.0f;
                    fz += __shfl_down_sync(0xffffffffu, fz, 16);
                    if (lane < 16) zp[f] = fz;
                }
                tc_fence_before();
                if (have) mbar_arrive(accfree + b);
                __threadfence();
                named_sync<128>(2);
                if (tid == 0) *slast = (atomicAdd(a.counters + a.B * a.H + bh, 1) == nruns - 1) ? 1 : 0;
                named_sync<128>(2);
                if (*slast) {
                    __threadfence();
                    ordered_sum4(a.dS_part + (size_t)bh * it.nchunk * C::D * C::DV, nruns, C::D * C::DV,
                                 a.dS_fin + (size_t)bh * C::D * C::DV, tid, 128);
                    ordered_sum4(a.dz_part + (size_t)bh * it.nchunk * C::D, nruns, C::D, a.dz_fin + (size_t)bh * C::D,
                                 tid, 128);
                    if (tid == 0) a.counters[a.B * a.H + bh] = 0;
                }
                named_sync<128>(2);
            }
            if (run_tiles > 0) ++ne;
            i0 = i1;
        }
        if (pend_g >= 0) dq_out(pend_g, pend_row);
        if (hacc.tiles > 0) hist_close(bins, hpart, a.lay.nint, hacc, tid, false, smax, warp, lane);
#pragma unroll
        for (int q = 0; q < C::PP; ++q) {
            float v = db_acc[q];
#pragma unroll
            for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
            if (lane == 0) atomicAdd(sdb + H * C::PP + q, v);
        }
        // dW^T accumulator (M = 64: input column cd in lane 32*(cd/16) + cd%16)
        if (warp < 4) {
            const int T = block_tiles(a, it);
            if (T > 0) wait_or_fail(wdone, 0, failed, status);
            tc_fence_after();
            uint32_t x[16];
            tmem_ld16(tbase + ((uint32_t)(warp << 5) << 16) + cW, x);
            tmem_wait_ld();
            const int cd = (warp << 4) | lane;
            if (T > 0 && lane < 16 && cd < C::d)
#pragma unroll
                for (int i = 0; i < C::MP; ++i) sdW[i * C::d + cd] = __uint_as_float(x[i]) + __uint_as_float(x[C::MP + i]);
        }
    }
    tc_fence_before();
    __syncthreads();
    store_param_partial<C>(a, sdW, sdb, a.gpart + (size_t)blockIdx.x * a.gsize);
    __syncthreads();
    if (warp == 0) tmem_dealloc(tbase, 512);
}

// ---------------------------------------------------------------------------
// key side

template <class C>
__global__ void __launch_bounds__(kBThreads, 1)
    k_tc_bwd_key_w(const __grid_constant__ CUtensorMap mapK, const __grid_constant__ CUtensorMap mapV, AttnArgs a,
                   int *status) {
    extern __shared__ uint8_t smem_raw[];
    const float fl = channel_floor(a.lay);  // lower bound of a channel output
    uint8_t *sm = align1024(smem_raw);
    constexpr int NS = C::NSK;
    constexpr uint32_t T16 = C::TILE;
    uint8_t *Sb = sm;                    // [NS] x (phi tile, K tile)
    uint8_t *Vb = Sb + NS * 2 * T16;     // V tile
    uint8_t *Gt = Vb + T16;              // [dU_hi | dU_lo | dU_hi | 0]
    uint8_t *Wop = Gt + T16;
    uint8_t *Wx = Wop + C::WOP;
    uint8_t *Sop = Wx + C::WXP;          // dV = phi [dS_hi; dS_lo]: rows per value column
    uint8_t *Sop2 = Sop + C::SOP;        // dphi = V [dS_hi; dS_lo]^T: rows per feature
    float *sTe = reinterpret_cast<float *>(Sop2 + C::SOP2);
    float *sAB = sTe + kEytzinger;
    float *sbias = sAB + kNint * 16;
    float *sdz = sbias + 32;
    int *bins = reinterpret_cast<int *>(sdz + C::D);
    float *sdW = reinterpret_cast<float *>(bins + kNint * 16);
    float *sdb = sdW + C::MP * C::d;
    float *smax = sdb + 16;
    uint64_t *bars = reinterpret_cast<uint64_t *>(smax + 2 * (kBWorkers / 32));
    uint64_t *fullk = bars;              // [NS]
    uint64_t *sfree = fullk + NS;        // [NS]
    uint64_t *fullv = sfree + NS;        // [1]
    uint64_t *vfree = fullv + 1;         // [1]
    uint64_t *uready = vfree + 1;        // [2]
    uint64_t *fready = uready + 2;       // [1] dphi in TMEM
    uint64_t *phiready = fready + 1;     // [1] count 512
    uint64_t *dvready = phiready + 1;    // [1]
    uint64_t *dvfree = dvready + 1;      // [1] count 512
    uint64_t *gready = dvfree + 1;       // [1] count 512
    uint64_t *gfree = gready + 1;        // [1]
    uint64_t *dkready = gfree + 1;       // [1]
    uint64_t *dkfree = dkready + 1;      // [1] count 512
    uint64_t *opready = dkfree + 1;      // [1] count 512
    uint64_t *wdone = opready + 1;       // [1]
    uint32_t *tslot = reinterpret_cast<uint32_t *>(wdone + 1);
    static_assert((2 * NS + 16) * 8 + 4 <= kBarBytes, "barrier area");

    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const Items it(a);
    // TMEM: U [2 x 32] | dphi [128] | dV [128] | dK [64] | dW (M = 64) [16]
    constexpr uint32_t cU = 0, cF = 64, cV = 192, cK = 320, cW = 384;

    if (tid == 0) {
        for (int i = 0; i < NS; ++i) { mbar_init(fullk + i, 1); mbar_init(sfree + i, 1); }
        mbar_init(fullv, 1); mbar_init(vfree, 1);
        for (int i = 0; i < 2; ++i) mbar_init(uready + i, 1);
        mbar_init(fready, 1); mbar_init(phiready, kBWorkers);
        mbar_init(dvready, 1); mbar_init(dvfree, kBWorkers);
        mbar_init(gready, kBWorkers); mbar_init(gfree, 1);
        mbar_init(dkready, 1); mbar_init(dkfree, kBWorkers);
        mbar_init(opready, kBWorkers); mbar_init(wdone, 1);
        fence_mbar_init();
    }
    if (warp == 0) { tmem_alloc(tslot, 512); tmem_relinquish(); }
    stage_phi_table<C>(a, sTe, sAB, sbias, Wop);
    stage_wx<C>(a, Wx, 0);
    for (int e = tid; e < kNint * 16; e += blockDim.x) bins[e] = 0;
    for (int e = tid; e < C::MP * C::d + 16; e += blockDim.x) sdW[e] = 0.0f;
    for (int e = tid; e < (int)(T16 / 16); e += blockDim.x) reinterpret_cast<uint4 *>(Gt)[e] = make_uint4(0, 0, 0, 0);
    float *hpart = a.gpart + (size_t)(gridDim.x + blockIdx.x) * a.gsize + C::MP * a.d + C::MP;
    for (int e = tid; e < a.lay.nint * 16; e += blockDim.x) hpart[e] = 0.0f;
    for (int item = it.begin; item < it.end && !a.padded_zeroed; ++item) {  // padded rows: zero gradients
        const ItemRange ir = item_range(a, it, item);
        __nv_bfloat16 *dK = static_cast<__nv_bfloat16 *>(a.dK) + head_rows(a, ir.bh) * C::d;
        __nv_bfloat16 *dV = static_cast<__nv_bfloat16 *>(a.dV) + head_rows(a, ir.bh) * C::DV;
        const int z0 = max(ir.r0, ir.r1);
        for (int e = tid; e < (ir.rend - z0) * C::d / 8; e += blockDim.x)
            reinterpret_cast<uint4 *>(dK + (size_t)z0 * C::d)[e] = make_uint4(0, 0, 0, 0);
        for (int e = tid; e < (ir.rend - z0) * C::DV / 8; e += blockDim.x)
            reinterpret_cast<uint4 *>(dV + (size_t)z0 * C::DV)[e] = make_uint4(0, 0, 0, 0);
    }
    fence_proxy_async_smem();
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tbase = *tslot;

    if (warp == kBTma) {
        if (lane < 2) {
            const int T = block_tiles(a, it);
            TileCursor cur;
            cur.start(a, it);
            bool failed = false;
            for (int g = 0; g < T && !failed; ++g, cur.next(a, it)) {
                if (lane == 0) {
                    const int s = g % NS;
                    if (g >= NS) wait_or_fail(sfree + s, ((g - NS) / NS) & 1, failed, status);
                    mbar_arrive_expect_tx(fullk + s, T16);
                    tma_load_3d(Sb + s * 2 * T16 + T16, &mapK, 0, cur.row0(), cur.g.bh, fullk + s);
                } else {
                    if (g >= 1) wait_or_fail(vfree, (g - 1) & 1, failed, status);
                    mbar_arrive_expect_tx(fullv, T16);
                    tma_load_3d(Vb, &mapV, 0, cur.row0(), cur.g.bh, fullv);
                }
            }
        }
    } else if (warp == kBMma) {
        if (lane == 0) {
            const int T = block_tiles(a, it);
            const uint64_t dS0 = sdesc(smem_u32(Sb), 16384, 1024, kSwizzle128);
            const uint64_t dV0 = sdesc(smem_u32(Vb), 16384, 1024, kSwizzle128);
            const uint64_t dG = sdesc(smem_u32(Gt), 16384, 1024, kSwizzle128);
            const uint64_t dWo = sdesc(smem_u32(Wop), 16, 1024, kSwizzle128);
            const uint64_t dWx = sdesc(smem_u32(Wx), 16, 1024, kSwizzle128);
            const uint64_t dSa = sdesc(smem_u32(Sop), 16, 1024, kSwizzle128);
            const uint64_t dSb = sdesc(smem_u32(Sop2), 16, 1024, kSwizzle128);
            bool failed = false;
            auto proj = [&](int g) {
                const int s = g % NS;
                wait_or_fail(fullk + s, (g / NS) & 1, failed, status);
                tc_fence_after();
                proj_mma<C>(tbase + cU + (g & 1) * C::NU, dadd(dS0, s * 2 * T16 + T16), dWo);
                mma_commit(uready + (g & 1));
            };
            auto fmma = [&](int g) {  // dphi = V [dS_hi; dS_lo]^T into the single dphi columns
                wait_or_fail(fullv, g & 1, failed, status);
                tc_fence_after();
                constexpr uint32_t idF = idesc_bf16(128, 2 * C::D, false, false);
#pragma unroll
                for (int k = 0; k < C::NKV; ++k)
                    mma_bf16_ss(tbase + cF, dadd(dV0, 32 * k), dadd(dSb, 32 * k), idF, k != 0);
                mma_commit(fready);
                mma_commit(vfree);
            };
            int op_phase = 0;
            if (T > 0) { proj(0); wait_or_fail(opready, op_phase++ & 1, failed, status); fmma(0); }
            if (T > 1) proj(1);
            TileCursor cur;
            cur.start(a, it);
            for (int g = 0; g < T && !failed; ++g) {
                const int s = g % NS;
                TileCursor nx = cur;
                nx.next(a, it);
                const bool next_new_run = (g + 1 < T) && nx.g.bh != cur.g.bh;
                // dV = phi [dS_hi; dS_lo]  (phi K-major over the D features)
                wait_or_fail(phiready, g & 1, failed, status);
                if (g >= 1) wait_or_fail(dvfree, (g - 1) & 1, failed, status);
                tc_fence_after();
                constexpr uint32_t idV = idesc_bf16(128, 2 * C::DV, false, false);
#pragma unroll
                for (int k = 0; k < C::D / 16; ++k)
                    mma_bf16_ss(tbase + cV, dadd(dS0, s * 2 * T16 + 32 * k), dadd(dSa, 32 * k), idV, k != 0);
                mma_commit(dvready);
                // dK = [dU_hi | dU_lo | dU_hi | 0] W and dW^T += K^T dU
                wait_or_fail(gready, g & 1, failed, status);
                if (g >= 1) wait_or_fail(dkfree, (g - 1) & 1, failed, status);
                tc_fence_after();
                constexpr uint32_t idK = idesc_bf16(128, C::d, false, false);
#pragma unroll
                for (int k = 0; k < 2; ++k) mma_bf16_ss(tbase + cK, dadd(dG, 32 * k), dadd(dWx, 32 * k), idK, k != 0);
                mma_commit(dkready);  // before the dW^T products: the workers read dK out sooner
                constexpr uint32_t idW = idesc_bf16(64, 16, true, true);
#pragma unroll
                for (int k = 0; k < 8; ++k)
                    mma_bf16_ss(tbase + cW, dadd(dS0, s * 2 * T16 + T16 + 2048 * k), dadd(dG, 2048 * k), idW,
                                (g > 0 || k > 0) ? 1u : 0u);
                mma_commit(gfree);
                mma_commit(sfree + s);
                // the workers have read dphi(g) (before gready): dphi of the next tile
                if (g + 1 < T) {
                    if (next_new_run) wait_or_fail(opready, op_phase++ & 1, failed, status);
                    fmma(g + 1);
                }
                if (g + 2 < T) proj(g + 2);
                cur = nx;
            }
            if (T > 0 && !failed) mma_commit(wdone);
            else mbar_arrive(wdone);
        }
    } else {
        const int H = warp >> 2, r = ((warp & 3) << 5) | lane;
        const uint32_t lrow = (uint32_t)((warp & 3) << 5) << 16;
        bool failed = false;
        float db_acc[C::PP];
#pragma unroll
        for (int q = 0; q < C::PP; ++q) db_acc[q] = 0.0f;
        HistAcc hacc;
        int g = 0;
        for (int i0 = it.begin; i0 < it.end;) {
            const int bh = i0 / it.nchunk;
            const int i1 = min(it.end, (bh + 1) * it.nchunk);
            int run_tiles = 0;
            for (int i = i0; i < i1; ++i) run_tiles += item_range(a, it, i).ntiles;
            if (run_tiles > 0) {
                named_sync<kBWorkers>(1);
                const float *dSg = a.dS_fin + (size_t)bh * C::D * C::DV;
                stage_rows_per_column<C>(dSg, Sop, tid, kBWorkers);
                stage_rows_per_feature<C>(dSg, Sop2, tid, kBWorkers);
                for (int e = tid; e < C::D; e += kBWorkers) sdz[e] = a.dz_fin[(size_t)bh * C::D + e];
                fence_proxy_async_smem();
                named_sync<kBWorkers>(1);
                mbar_arrive(opready);
            }
            __nv_bfloat16 *dK = static_cast<__nv_bfloat16 *>(a.dK) + head_rows(a, bh) * C::d;
            __nv_bfloat16 *dV = static_cast<__nv_bfloat16 *>(a.dV) + head_rows(a, bh) * C::DV;
            for (int item = i0; item < i1; ++item) {
                const ItemRange ir = item_range(a, it, item);
                for (int t = 0; t < ir.ntiles; ++t, ++g) {
                    const int s = g % NS;
                    const int row0 = ir.r0 + t * 128;
                    const int nvalid = min(128, ir.r1 - row0);
                    const bool valid = r < nvalid;
                    uint8_t *phit = Sb + s * 2 * T16, *kt = phit + T16;
                    wait_or_fail(uready + (g & 1), (g >> 1) & 1, failed, status);
                    tc_fence_after();
                    float u[C::PP];
                    int j[C::PP];
                    {
                        static_assert(C::PP == 2, "two projections per thread");
                        uint32_t xh[2], xm[2], xl[2];
                        const uint32_t ucol = tbase + lrow + cU + (g & 1) * C::NU + H * C::PP;
                        tmem_ld2(ucol, xh);
                        tmem_ld2(ucol + C::MP, xm);
                        tmem_ld2(ucol + 2 * C::MP, xl);
                        tmem_wait_ld();
#pragma unroll
                        for (int q = 0; q < C::PP; ++q)
                            u[q] = (__uint_as_float(xh[q]) + __uint_as_float(xm[q])) + __uint_as_float(xl[q]) +
                                   sbias[H * C::PP + q];
                    }
                    search<C::PP>(sTe, u, j);
#pragma unroll
                    for (int q = 0; q < C::PP; ++q) {
                        float al[8], y[8];
                        channel_eval(sAB, j[q], u[q], fl, al, y);
                        *reinterpret_cast<uint4 *>(phit + sw128_chunk(r, H * C::PP + q)) =
                            valid ? pack8(y) : make_uint4(0, 0, 0, 0);
                    }
                    if (!valid && H == 0) zero_row(kt, r);
                    fence_proxy_async_smem();
                    tc_fence_before();
                    mbar_arrive(phiready);
                    // dphi(k) = dS v + dz  ->  dU, histogram
                    wait_or_fail(fready, g & 1, failed, status);
                    tc_fence_after();
                    bool hon = hacc.open;
                    float dU[C::PP], gv[C::PP][8];
#pragma unroll
                    for (int q = 0; q < C::PP; ++q) {
                        const int i = H * C::PP + q;
                        float al[8], y[8];
                        channel_eval(sAB, j[q], u[q], fl, al, y);
                        uint32_t ph[8], pl[8];
                        tmem_ld8(tbase + lrow + cF + 8 * i, ph);
                        tmem_ld8(tbase + lrow + cF + C::D + 8 * i, pl);
                        tmem_wait_ld();
                        float du = 0.0f;
#pragma unroll
                        for (int l = 0; l < 8; ++l) {
                            const float dphi = __uint_as_float(ph[l]) + __uint_as_float(pl[l]) + sdz[8 * i + l];
                            const float gl = (valid && y[l] > fl) ? dphi : 0.0f;
                            gv[q][l] = gl;
                            du = fmaf(gl, al[l], du);
                        }
                        dU[q] = du;
                        db_acc[q] += du;
                    }
                    if (g >= 1) wait_or_fail(gfree, (g - 1) & 1, failed, status);
                    {
                        uint32_t vh, vl;
                        dU_pack(dU, vh, vl);
                        *reinterpret_cast<uint32_t *>(Gt + sw128_chunk(r, 0) + H * 4) = vh;
                        *reinterpret_cast<uint32_t *>(Gt + sw128_chunk(r, 1) + H * 4) = vl;
                        *reinterpret_cast<uint32_t *>(Gt + sw128_chunk(r, 2) + H * 4) = vh;
                    }
                    fence_proxy_async_smem();
                    tc_fence_before();
                    mbar_arrive(gready);
                    if (!hon) {  // first tile with a nonzero g in the block: its maxima give the first scales
                        float m0 = 0.0f, m1 = 0.0f;
#pragma unroll
                        for (int q = 0; q < C::PP; ++q)
#pragma unroll
                            for (int l = 0; l < 8; ++l) {
                                m0 = finite_max(m0, gv[q][l]);
                                m1 = finite_max(m1, gv[q][l] * u[q]);
                            }
                        hon = hist_open(hacc, m0, m1, smax, warp, lane);
                    }
                    if (hon) {
                        hist_add<C::PP>(bins, hpart, hacc, j, u, gv, dU);
                        if (++hacc.tiles == hist_tiles<C::MP>()) hist_close(bins, hpart, a.lay.nint, hacc, tid, true, smax, warp, lane);
                    }
                    // dV = hi + lo
                    wait_or_fail(dvready, g & 1, failed, status);
                    tc_fence_after();
                    {
                        const uint32_t vcol = tbase + lrow + cV + H * 16;
                        uint32_t xh[16], xl[16];
                        tmem_ld16(vcol, xh);
                        tmem_ld16(vcol + C::DV, xl);
                        tmem_wait_ld();
                        tc_fence_before();
                        mbar_arrive(dvfree);
                        if (valid) {
                            float f0[8], f1[8];
#pragma unroll
                            for (int c = 0; c < 8; ++c) {
                                f0[c] = __uint_as_float(xh[c]) + __uint_as_float(xl[c]);
                                f1[c] = __uint_as_float(xh[8 + c]) + __uint_as_float(xl[8 + c]);
                            }
                            uint4 *dst = reinterpret_cast<uint4 *>(dV + (size_t)(row0 + r) * C::DV + H * 16);
                            dst[0] = pack8(f0);
                            dst[1] = pack8(f1);
                        }
                    }
                    // dK
                    wait_or_fail(dkready, g & 1, failed, status);
                    tc_fence_after();
                    {
                        uint32_t x[16];
                        tmem_ld16(tbase + lrow + cK + H * 16, x);
                        tmem_wait_ld();
                        tc_fence_before();
                        mbar_arrive(dkfree);
                        if (valid) {
                            float f0[8], f1[8];
#pragma unroll
                            for (int c = 0; c < 8; ++c) { f0[c] = __uint_as_float(x[c]); f1[c] = __uint_as_float(x[8 + c]); }
                            uint4 *dst = reinterpret_cast<uint4 *>(dK + (size_t)(row0 + r) * C::d + H * 16);
                            dst[0] = pack8(f0);
                            dst[1] = pack8(f1);
                        }
                    }
                }
            }
            i0 = i1;
        }
        if (hacc.tiles > 0) hist_close(bins, hpart, a.lay.nint, hacc, tid, false, smax, warp, lane);
#pragma unroll
        for (int q = 0; q < C::PP; ++q) {
            float v = db_acc[q];
#pragma unroll
            for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
            if (lane == 0) atomicAdd(sdb + H * C::PP + q, v);
        }
        if (warp < 4) {  // dW^T accumulator (M = 64: input column cd in lane 32*(cd/16) + cd%16)
            const int T = block_tiles(a, it);
            if (T > 0) wait_or_fail(wdone, 0, failed, status);
            tc_fence_after();
            uint32_t x[16];
            tmem_ld16(tbase + ((uint32_t)(warp << 5) << 16) + cW, x);
            tmem_wait_ld();
            const int cd = (warp << 4) | lane;
            if (T > 0 && lane < 16 && cd < C::d)
#pragma unroll
                for (int i = 0; i < C::MP; ++i) sdW[i * C::d + cd] = __uint_as_float(x[i]) + __uint_as_float(x[C::MP + i]);
        }
    }
    tc_fence_before();
    __syncthreads();
    store_param_partial<C>(a, sdW, sdb, a.gpart + (size_t)(gridDim.x + blockIdx.x) * a.gsize);
    __syncthreads();
    if (warp == 0) tmem_dealloc(tbase, 512);
}

}  // namespace

bool tc_make_map(CUtensorMap *m, const void *base, int width, int n, int BH, int hs_mul);

cudaError_t launch_tc_bwd_wide(const AttnArgs &a0, bool have_stats, cudaStream_t s) {
    using C = B64;
    cudaError_t e;
    const AttnArgs a = tc_balanced_items(a0, s, &e, 2 | 4 | 8);  // dQ, dK, dV
    if (e != cudaSuccess) return e;
    const int grid = tc_grid(a);
    if (!have_stats && (e = launch_tc_stats(a, s)) != cudaSuccess) return e;
    CUtensorMap mQ, mdO, mK, mV;
    if (!tc_make_map(&mQ, a.Q, a.d, a.n, a.B * a.H, a.hs_mul) ||
        !tc_make_map(&mdO, a.dO, a.dv, a.n, a.B * a.H, a.hs_mul) ||
        !tc_make_map(&mK, a.K, a.d, a.n, a.B * a.H, a.hs_mul) || !tc_make_map(&mV, a.V, a.dv, a.n, a.B * a.H, a.hs_mul))
        return cudaErrorInvalidValue;
    if ((e = cudaFuncSetAttribute(k_tc_bwd_query_w<C>, cudaFuncAttributeMaxDynamicSharedMemorySize, C::SMEM_Q)) !=
        cudaSuccess)
        return e;
    if ((e = cudaFuncSetAttribute(k_tc_bwd_key_w<C>, cudaFuncAttributeMaxDynamicSharedMemorySize, C::SMEM_K)) !=
        cudaSuccess)
        return e;
    int *st = reinterpret_cast<int *>(reinterpret_cast<char *>(a.counters) - 256);
    LUNA_LAUNCH("tc_bwd_query", k_tc_bwd_query_w<C>, grid, kBThreads, C::SMEM_Q, s, mQ, mdO, a, st);
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
    if ((e = launch_chrms_dstate(a, s)) != cudaSuccess) return e;
    LUNA_LAUNCH("tc_bwd_key", k_tc_bwd_key_w<C>, grid, kBThreads, C::SMEM_K, s, mK, mV, a, st);
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
    int nparts = 0;
    if ((e = launch_chrms_backward(a, 2 * grid, &nparts, s)) != cudaSuccess) return e;
    return launch_grad_reduce(a, nparts, s);
}

}  // namespace luna
