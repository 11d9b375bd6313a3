// Tensor-core (tcgen05 / TMEM / TMA) kernels for bf16 I/O on sm_103a.
//
// Persistent kernels: one block per SM walks a contiguous range of work items
// (head, chunk of 128-row tiles).  Warp roles in a block of 576 threads:
//   warps 0..15  workers, four per row: warps w, w+4, w+8, w+12 own TMEM lanes
//                32*(w%4)..+31 and each evaluates the feature map for a
//                quarter of the M projections of those rows;
//   warp 16      TMA: lane 0 streams the X (query / key) tiles, lane 1 the V
//                tiles, each into its own ring of shared-memory stages;
//   warp 17      MMA: lane 0 issues every tcgen05.mma and commits it to the
//                mbarriers that release stages and wake the workers.
//
// Forward key pass per tile (Sec. 4, S_KV and S_K1):
//   MMA  U = K [W_hi; W_lo]^T                      (projections -> TMEM)
//   workers: u = U_hi + U_lo + b; interval j of u from the bucketed search
//            block; phi = relu(alpha_j u + beta_j) for the 8 channels, written
//            as bf16 hi and lo tiles; z += phi in fp32 registers
//   MMA  S += [phi_hi | phi_lo]^T V                 (MN-major operands)
// Forward query pass (Eq. kernel-attn):
//   MMA U, workers phi(Q) (bf16) and the fp32 normaliser phi.z,
//   MMA  num = phi [S_hi; S_lo]^T,  O = num / (phi.z + eps)
// S and W enter their products split into bf16 hi + lo parts.
#include <atomic>

#include "luna_tc_dev.cuh"

namespace luna {
namespace {
using namespace sm100;
using namespace simt;
using namespace tcdev;

constexpr int kWorkerWarps = 16;
constexpr int kWorkers = kWorkerWarps * 32;
constexpr int kTmaWarp = 16, kMmaWarp = 17;
constexpr int kThreadsTC = kWorkers + 64;

template <int DX_, int DV_, int MP_>
struct Cfg {
    static constexpr int DX = DX_;                // X tile columns (d rounded up to 64)
    static constexpr int DV = DV_;                // value width
    static constexpr int MP = MP_;                // projections
    static constexpr int D = MP * 8;              // features (L = 8)
    static constexpr int KBX = DX / 64;           // 64-column blocks of an X tile
    static constexpr int VC = DV < 64 ? 64 : DV;  // V tile columns (zero padded)
    static constexpr int NVB = VC / 64;
    static constexpr int NPB = D / 64;            // 64-feature blocks of a phi tile
    static constexpr int NU = 2 * MP;             // projection columns (hi, lo)
    static constexpr int PP = MP / 4;             // projections per worker thread
    static constexpr bool MERGE = (D == 64);      // phi_hi and phi_lo stacked into one M = 128 operand
    static constexpr uint32_t XT = 128u * DX * 2;
    static constexpr uint32_t VT = 128u * VC * 2;
    static constexpr uint32_t PT = 128u * D * 2;  // one bf16 phi tile
    static constexpr uint32_t WOP = (uint32_t)NU * DX * 2;
    static constexpr uint32_t TABLE = (kEytzinger + kNint * 16 + 32) * 4;
    static constexpr uint32_t MISC = 1024;
    static constexpr bool SMALL = XT <= 16384 && VT <= 16384;
    // key pass
    static constexpr int NX_K = SMALL ? 3 : 2;
    static constexpr int NV_K = SMALL ? 3 : 1;
    static constexpr int NP_K = SMALL ? 2 : 1;
    static constexpr uint32_t ZPART = 4u * D * 4;
    static constexpr uint32_t SSTAGE = MERGE ? 64u * DV * 4 : 0u;
    static constexpr uint32_t FIX_K = WOP + TABLE + ZPART + SSTAGE + MISC + 1024;
    static constexpr uint32_t SMEM_K = NX_K * XT + NV_K * VT + NP_K * 2 * PT + FIX_K;
    static constexpr int TMEM_K_USED = 2 * NU + 2 * DV;
    static constexpr int TMEM_K = TMEM_K_USED <= 64 ? 64 : TMEM_K_USED <= 128 ? 128 : TMEM_K_USED <= 256 ? 256 : 512;
    // query pass
    static constexpr uint32_t SOP = 2u * DV * D * 2;  // [S_hi; S_lo]^T operand
    static constexpr int NP_Q = SMALL ? 2 : 1;
    static constexpr int NX_Q = SMALL ? 4 : 2;
    static constexpr uint32_t FIX_Q = WOP + SOP + TABLE + D * 4 + 2 * 4 * 128 * 4 + MISC + 1024;
    static constexpr uint32_t SMEM_Q = NX_Q * XT + NP_Q * PT + FIX_Q;
    static constexpr int NN_Q = (2 * NU + 4 * DV <= 256) ? 2 : 1;
    static constexpr int TMEM_Q_USED = 2 * NU + 2 * DV * NN_Q;
    static constexpr int TMEM_Q = TMEM_Q_USED <= 64 ? 64 : TMEM_Q_USED <= 128 ? 128 : TMEM_Q_USED <= 256 ? 256 : 512;
    static_assert(SMEM_K <= kSmemLimit && SMEM_Q <= kSmemLimit, "shared memory budget");
    static_assert(TMEM_K_USED <= 512 && TMEM_Q_USED <= 512, "tensor memory budget");
    static_assert(PP == 2 || PP == 4, "projections per worker");
};

// Worker: phi for projections [Q*PP, Q*PP+PP) of row r from the projection
// columns in TMEM.  The PP interval searches run interleaved over the
// bucketed search block (j = the number of kinks strictly below u).
// Writes the bf16 chunks of the phi tile (and, if plo is not null, the bf16
// residual phi - bf16(phi) into a second tile), zeros for rows that are not
// valid.  Optionally adds phi into zacc (fp32 feature sums) and accumulates the
// fp32 normaliser phi . z.
template <class C>
__device__ __forceinline__ void phi_row_quarter(int Q, uint32_t tmem_u_row, const float *sTe, const float *sAB,
                                                const float *sbias, float fl, bool valid, int r, uint8_t *phi,
                                                uint8_t *plo,
                                                float *zacc, const float *sz, float &den) {
    constexpr int PP = C::PP;
    float u[PP];
    {
        // this thread's PP projections: hi parts at columns Q*PP.., lo parts MP columns further
        uint32_t xh[PP], xl[PP];
        if constexpr (PP == 2) {
            tmem_ld2(tmem_u_row + Q * PP, xh);
            tmem_ld2(tmem_u_row + C::MP + Q * PP, xl);
        } else {
            tmem_ld4(tmem_u_row + Q * PP, xh);
            tmem_ld4(tmem_u_row + C::MP + Q * PP, xl);
        }
        tmem_wait_ld();
#pragma unroll
        for (int q = 0; q < PP; ++q) u[q] = __uint_as_float(xh[q]) + __uint_as_float(xl[q]);
    }
#pragma unroll
    for (int q = 0; q < PP; ++q) u[q] += sbias[Q * PP + q];
    int node[PP];
    search_bucketed<PP>(sTe, u, node);
#pragma unroll
    for (int q = 0; q < PP; ++q) {
        const int i = Q * PP + q;
        uint4 ph = make_uint4(0u, 0u, 0u, 0u), pl = make_uint4(0u, 0u, 0u, 0u);
        if (valid) {
            const int j = node[q];
            const float4 *ab = reinterpret_cast<const float4 *>(sAB);
            float y[8];
#pragma unroll
            for (int k = 0; k < 4; ++k) {
                const float4 v = ab[ab_slot(j, k)];
                y[2 * k] = fmaxf(fmaf(v.x, u[q], v.y), fl);
                y[2 * k + 1] = fmaxf(fmaf(v.z, u[q], v.w), fl);
            }
            if (zacc) {
#pragma unroll
                for (int l = 0; l < 8; ++l) zacc[q * 8 + l] += y[l];
            }
            if (sz) {
#pragma unroll
                for (int l = 0; l < 8; ++l) den = fmaf(y[l], sz[i * 8 + l], den);
            }
            uint32_t hw[4], lw[4];
#pragma unroll
            for (int k = 0; k < 4; ++k) {
                const __nv_bfloat162 hb = __floats2bfloat162_rn(y[2 * k], y[2 * k + 1]);
                hw[k] = *reinterpret_cast<const uint32_t *>(&hb);
                if (plo) lw[k] = pack_bf16x2(y[2 * k] - __low2float(hb), y[2 * k + 1] - __high2float(hb));
            }
            ph = make_uint4(hw[0], hw[1], hw[2], hw[3]);
            if (plo) pl = make_uint4(lw[0], lw[1], lw[2], lw[3]);
        }
        const uint32_t off = (i / 8) * 16384 + sw128_chunk(r, i % 8);
        *reinterpret_cast<uint4 *>(phi + off) = ph;
        if (plo) *reinterpret_cast<uint4 *>(plo + off) = pl;
    }
}

// Projection MMA of tile g into TMEM stage g & 1.
template <class C>
__device__ __forceinline__ void issue_proj(uint32_t tmem_u, uint64_t dx, uint64_t dw) {
    constexpr uint32_t idesc = idesc_bf16(128, C::NU, false, false);
#pragma unroll
    for (int kb = 0; kb < C::KBX; ++kb)
#pragma unroll
        for (int k = 0; k < 4; ++k)
            mma_bf16_ss(tmem_u, dadd(dx, kb * 16384 + 32 * k), dadd(dw, kb * (C::NU * 128) + 32 * k), idesc,
                        (kb | k) != 0);
}

// ---------------------------------------------------------------------------
// forward key pass: S_KV = phi(K)^T V and S_K1 = phi(K)^T 1 per (head, chunk)
//
// phi(K) enters the contraction as bf16 hi + lo tiles so that the key
// statistics carry ~16 significant bits of phi (the backward pass subtracts
// nearly equal terms built from S and z); z is summed by the workers in fp32.
// Each run's statistics go to its partial slot; the last run of a head to
// finish sums the partials in order (warps 0..3 only, so that the pipeline
// keeps running).  Per-item mode (the state segments of the streaming form,
// a.seg_S set): every item is its own run, its statistics go to slot
// (head, item), and nothing is summed here.

template <class C>
__global__ void __launch_bounds__(kThreadsTC, 1)
    k_tc_keys(const __grid_constant__ CUtensorMap mapK, const __grid_constant__ CUtensorMap mapV, AttnArgs a,
              int *status) {
    extern __shared__ uint8_t smem_raw[];
    uint8_t *sm = align1024(smem_raw);
    constexpr int NX = C::NX_K, NV = C::NV_K, NP = C::NP_K;
    uint8_t *Xb = sm;
    uint8_t *Vb = Xb + NX * C::XT;
    uint8_t *Pb = Vb + NV * C::VT;  // [NP][hi, lo]
    uint8_t *Wop = Pb + NP * 2 * C::PT;
    float *sTe = reinterpret_cast<float *>(Wop + C::WOP);
    float *sAB = sTe + kEytzinger;
    float *sbias = sAB + kNint * 16;
    float *zpart = sbias + 32;         // [4][D]
    float *sstage = zpart + 4 * C::D;  // [64][DV] (stacked operand only)
    uint64_t *bars = reinterpret_cast<uint64_t *>(sstage + C::SSTAGE / 4);
    uint64_t *fullx = bars;            // [NX] X tile landed
    uint64_t *xfree = fullx + NX;      // [NX] projection MMA consumed it
    uint64_t *fullv = xfree + NX;      // [NV] V tile landed
    uint64_t *vfree = fullv + NV;      // [NV] contraction consumed it
    uint64_t *uready = vfree + NV;     // [2] projection in TMEM
    uint64_t *phiready = uready + 2;   // [NP] workers wrote phi (count 512)
    uint64_t *pfree = phiready + NP;   // [NP] contraction consumed phi
    uint64_t *accdone = pfree + NP;    // [2] item statistics complete
    uint64_t *accfree = accdone + 2;   // [2] item statistics read (count 128)
    uint32_t *tslot = reinterpret_cast<uint32_t *>(accfree + 2);
    int *slast = reinterpret_cast<int *>(tslot + 1);

    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const bool per_item = a.seg_S != nullptr;

    if (tid == 0) {
        for (int i = 0; i < NX; ++i) { mbar_init(fullx + i, 1); mbar_init(xfree + i, 1); }
        for (int i = 0; i < NV; ++i) { mbar_init(fullv + i, 1); mbar_init(vfree + i, 1); }
        for (int i = 0; i < 2; ++i) mbar_init(uready + i, 1);
        for (int i = 0; i < NP; ++i) { mbar_init(phiready + i, kWorkers); mbar_init(pfree + i, 1); }
        for (int i = 0; i < 2; ++i) { mbar_init(accdone + i, 1); mbar_init(accfree + i, 128); }
        fence_mbar_init();
    }
    if (warp == 0) { tmem_alloc(tslot, C::TMEM_K); tmem_relinquish(); }
    stage_phi_table<C>(a, sTe, sAB, sbias, Wop);
    grid_dependency_sync();  // the work split and the counters are read from here on
    const Items it(a);
    fence_proxy_async_smem();
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tbase = *tslot;
    const uint32_t tmem_acc = tbase + 2 * C::NU;  // [2] x DV cols

    if (warp == kTmaWarp) {
        if (lane < 2) {
            const int T = block_tiles(a, it);
            TileCursor cur;
            cur.start(a, it);
            bool failed = false;
            for (int g = 0; g < T && !failed; ++g, cur.next(a, it)) {
                if (lane == 0) {
                    const int x = g % NX;
                    if (g >= NX) wait_or_fail(xfree + x, ((g - NX) / NX) & 1, failed, status);
                    mbar_arrive_expect_tx(fullx + x, C::XT);
                    for (int kb = 0; kb < C::KBX; ++kb)
                        tma_load_3d(Xb + x * C::XT + kb * 16384, &mapK, kb * 64, cur.row0(), cur.g.bh, fullx + x);
                } else {
                    const int v = g % NV;
                    if (g >= NV) wait_or_fail(vfree + v, ((g - NV) / NV) & 1, failed, status);
                    mbar_arrive_expect_tx(fullv + v, C::VT);
                    for (int vb = 0; vb < C::NVB; ++vb)
                        tma_load_3d(Vb + v * C::VT + vb * 16384, &mapV, vb * 64, cur.row0(), cur.g.bh, fullv + v);
                }
                if (g + 1 < T) {  // the next tile into L2 while this one is worked on
                    TileCursor nx = cur;
                    nx.next(a, it);
                    if (lane == 0)
                        for (int kb = 0; kb < C::KBX; ++kb) tma_prefetch_3d(&mapK, kb * 64, nx.row0(), nx.g.bh);
                    else
                        for (int vb = 0; vb < C::NVB; ++vb) tma_prefetch_3d(&mapV, vb * 64, nx.row0(), nx.g.bh);
                }
            }
        }
    } else if (warp == kMmaWarp) {
        if (lane == 0) {
            const int T = block_tiles(a, it);
            const uint64_t dx0 = sdesc(smem_u32(Xb), 16, 1024, kSwizzle128);
            const uint64_t dw0 = sdesc(smem_u32(Wop), 16, 1024, kSwizzle128);
            const uint64_t dp0 = sdesc(smem_u32(Pb), 16384, 1024, kSwizzle128);
            const uint64_t dv0 = sdesc(smem_u32(Vb), 16384, 1024, kSwizzle128);
            bool failed = false;
            auto proj = [&](int g) {
                const int x = g % NX;
                wait_or_fail(fullx + x, (g / NX) & 1, failed, status);
                tc_fence_after();
                issue_proj<C>(tbase + (g & 1) * C::NU, dadd(dx0, x * C::XT), dw0);
                mma_commit(uready + (g & 1));
                mma_commit(xfree + x);
            };
            if (T > 0) proj(0);
            if (T > 1) proj(1);
            // runs: maximal stretches of this block's items that share a head; S accumulates over a run
            int g = 0, ne = 0;
            for (int i0 = it.begin; i0 < it.end && !failed;) {
                const int bh = i0 / it.nchunk;
                const int i1 = per_item ? i0 + 1 : min(it.end, (bh + 1) * it.nchunk);
                int run_tiles = 0;
                for (int i = i0; i < i1; ++i) run_tiles += item_range(a, it, i).ntiles;
                if (run_tiles > 0) {
                    const int b = ne & 1;
                    if (ne >= 2) wait_or_fail(accfree + b, ((ne - 2) >> 1) & 1, failed, status);
                    const uint32_t tmem_s = tmem_acc + b * C::DV;
                    for (int t = 0; t < run_tiles && !failed; ++t, ++g) {
                        const int p = g % NP, v = g % NV;
                        wait_or_fail(phiready + p, (g / NP) & 1, failed, status);
                        wait_or_fail(fullv + v, (g / NV) & 1, failed, status);
                        tc_fence_after();
                        const uint64_t ph = dadd(dp0, p * 2 * C::PT), bv = dadd(dv0, v * C::VT);
                        constexpr uint32_t idS = idesc_bf16(128, C::DV, true, true);
#pragma unroll
                        for (int k = 0; k < 8; ++k) {
                            const uint32_t acc = (t > 0 || k > 0) ? 1u : 0u;
                            // stacked operand: rows 0..63 of A are phi_hi, rows 64..127 phi_lo (+16 KB)
                            mma_bf16_ss(tmem_s, dadd(ph, 2048 * k), dadd(bv, 2048 * k), idS, acc);
                            if constexpr (!C::MERGE)
                                mma_bf16_ss(tmem_s, dadd(ph, C::PT + 2048 * k), dadd(bv, 2048 * k), idS, 1u);
                        }
                        mma_commit(pfree + p);
                        mma_commit(vfree + v);
                        if (t == run_tiles - 1) mma_commit(accdone + b);
                        if (g + 2 < T) proj(g + 2);
                    }
                    ++ne;
                }
                i0 = i1;
            }
        }
    } else {
        const int Q = warp >> 2, r = ((warp & 3) << 5) | lane;
        const uint32_t lrow = (uint32_t)((warp & 3) << 5) << 16;
        float zacc[C::PP * 8];
#pragma unroll
        for (int k = 0; k < C::PP * 8; ++k) zacc[k] = 0.0f;
        float dummy = 0.0f;
        bool failed = false;
        int g = 0, ne = 0;
        for (int i0 = it.begin; i0 < it.end;) {
            const int bh = i0 / it.nchunk;
            const int i1 = per_item ? i0 + 1 : min(it.end, (bh + 1) * it.nchunk);
            int run_tiles = 0;
            for (int item = i0; item < i1; ++item) {
                const ItemRange ir = item_range(a, it, item);
                run_tiles += ir.ntiles;
                for (int t = 0; t < ir.ntiles; ++t, ++g) {
                    const int p = g % NP, v = g % NV;
                    const int nvalid = min(128, ir.r1 - (ir.r0 + t * 128));
                    wait_or_fail(uready + (g & 1), (g >> 1) & 1, failed, status);
                    if (g >= NP) wait_or_fail(pfree + p, ((g - NP) / NP) & 1, failed, status);
                    tc_fence_after();
                    uint8_t *ph = Pb + p * 2 * C::PT, *pl = ph + C::PT;
                    const bool valid = r < nvalid;
                    phi_row_quarter<C>(Q, tbase + lrow + (g & 1) * C::NU, sTe, sAB, sbias, channel_floor(a.lay), valid, r, ph, pl, zacc,
                                   nullptr, dummy);
                    if (!valid && Q == 0) {  // padded rows: clear V so that no garbage enters S
                        wait_or_fail(fullv + v, (g / NV) & 1, failed, status);
                        uint8_t *vrow = Vb + v * C::VT;
#pragma unroll
                        for (int vb = 0; vb < C::NVB; ++vb)
#pragma unroll
                            for (int c = 0; c < 8; ++c)
                                *reinterpret_cast<uint4 *>(vrow + vb * 16384 + sw128_chunk(r, c)) =
                                    make_uint4(0, 0, 0, 0);
                    }
                    fence_proxy_async_smem();
                    tc_fence_before();
                    mbar_arrive(phiready + p);
                }
            }
            // z of this run: sum the 128 rows of each warp group, then over the four row groups.  The
            // first barrier keeps these writes behind the previous run's epilogue (warps 0..3 read zpart
            // there while the other workers may already have finished a run without tiles).
#pragma unroll
            for (int k = 0; k < C::PP * 8; ++k) {
                float v = zacc[k];
#pragma unroll
                for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
                zacc[k] = v;
            }
            named_sync<kWorkers>(1);
#pragma unroll
            for (int k = 0; k < C::PP * 8; ++k) {
                if (lane == 0) zpart[(warp & 3) * C::D + Q * C::PP * 8 + k] = zacc[k];
                zacc[k] = 0.0f;
            }
            named_sync<kWorkers>(1);
            if (warp < 4) {
                // run epilogue: statistics of this block's part of head bh -> its partial slot
                const RunSlot rs = run_slot(a, it, bh);
                const int nruns = rs.nruns;
                const size_t slot = per_item ? (size_t)i0 : (size_t)bh * it.nchunk + rs.rank;
                float *Sp = a.S_part + slot * C::D * C::DV;
                float *zp = a.z_part + slot * C::D;
                const int row = (warp << 5) | lane;
                const uint32_t lrow0 = (uint32_t)(warp << 5) << 16;
                const bool have = run_tiles > 0;
                const int b = ne & 1;
                if (have) wait_or_fail(accdone + b, (ne >> 1) & 1, failed, status);
                tc_fence_after();
                const uint32_t tmem_s = tmem_acc + b * C::DV;
                // accumulator rows: feature f, and (stacked operand) the lo part of feature f at row 64 + f
                const int f = C::MERGE ? (row & 63) : row;
                if (C::MERGE && row >= 64) {
#pragma unroll
                    for (int c0 = 0; c0 < C::DV; c0 += 16) {
                        uint32_t x[16];
                        if (have) { tmem_ld16(lrow0 + tmem_s + c0, x); tmem_wait_ld(); }
#pragma unroll
                        for (int c = 0; c < 16; ++c) sstage[f * C::DV + c0 + c] = have ? __uint_as_float(x[c]) : 0.0f;
                    }
                }
                if constexpr (C::MERGE) named_sync<128>(2);
                if (!C::MERGE || row < 64) {
#pragma unroll
                    for (int c0 = 0; c0 < C::DV; c0 += 16) {
                        uint32_t x[16];
                        if (have) { tmem_ld16(lrow0 + tmem_s + c0, x); tmem_wait_ld(); }
#pragma unroll
                        for (int c = 0; c < 16; c += 4) {
                            float4 o;
                            o.x = have ? __uint_as_float(x[c]) : 0.0f;
                            o.y = have ? __uint_as_float(x[c + 1]) : 0.0f;
                            o.z = have ? __uint_as_float(x[c + 2]) : 0.0f;
                            o.w = have ? __uint_as_float(x[c + 3]) : 0.0f;
                            if (C::MERGE) {
                                o.x += sstage[f * C::DV + c0 + c];
                                o.y += sstage[f * C::DV + c0 + c + 1];
                                o.z += sstage[f * C::DV + c0 + c + 2];
                                o.w += sstage[f * C::DV + c0 + c + 3];
                            }
                            *reinterpret_cast<float4 *>(Sp + f * C::DV + c0 + c) = o;
                        }
                    }
                    zp[f] = zpart[f] + zpart[C::D + f] + zpart[2 * C::D + f] + zpart[3 * C::D + f];
                }
                tc_fence_before();
                if (have) mbar_arrive(accfree + b);
                // the last block of this head to finish sums the partials in block order
                __threadfence();
                named_sync<128>(2);
                if (tid == 0) *slast = (!per_item && atomicAdd(a.counters + bh, 1) == nruns - 1) ? 1 : 0;
                named_sync<128>(2);
                if (*slast) {
                    __threadfence();
                    ordered_sum4(a.S_part + (size_t)bh * it.nchunk * C::D * C::DV, nruns, C::D * C::DV,
                                 a.S_fin + head_state(a, bh) * C::D * C::DV, tid, 128);
                    ordered_sum4(a.z_part + (size_t)bh * it.nchunk * C::D, nruns, C::D, a.z_fin + head_state(a, bh) * C::D,
                                 tid, 128);
                    if (tid == 0) a.counters[bh] = 0;
                }
                named_sync<128>(2);
            }
            if (run_tiles > 0) ++ne;
            i0 = i1;
        }
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 0) tmem_dealloc(tbase, C::TMEM_K);
}

// ---------------------------------------------------------------------------
// forward query pass: O = phi(Q) S / (phi(Q).z + eps)

template <class C>
__global__ void __launch_bounds__(kThreadsTC, 1)
    k_tc_query(const __grid_constant__ CUtensorMap mapQ, AttnArgs a, int *status) {
    extern __shared__ uint8_t smem_raw[];
    uint8_t *sm = align1024(smem_raw);
    constexpr int NX = C::NX_Q, NP = C::NP_Q, NN = C::NN_Q;
    uint8_t *Xb = sm;
    uint8_t *Pb = Xb + NX * C::XT;
    uint8_t *Wop = Pb + NP * C::PT;
    uint8_t *Sop = Wop + C::WOP;
    float *sTe = reinterpret_cast<float *>(Sop + C::SOP);
    float *sAB = sTe + kEytzinger;
    float *sbias = sAB + kNint * 16;
    float *sz = sbias + 32;
    float *sden = sz + C::D;  // [2 tiles][4 quarters][128 rows]
    uint64_t *bars = reinterpret_cast<uint64_t *>(sden + 1024);
    uint64_t *fullx = bars;               // [NX]
    uint64_t *xfree = fullx + NX;         // [NX]
    uint64_t *uready = xfree + NX;        // [2]
    uint64_t *phiready = uready + 2;      // [NP] count 512
    uint64_t *pfree = phiready + NP;      // [NP]
    uint64_t *numready = pfree + NP;      // [NN]
    uint64_t *numfree = numready + NN;    // [NN] count 512
    uint32_t *tslot = reinterpret_cast<uint32_t *>(numfree + NN);

    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;

    if (tid == 0) {
        for (int i = 0; i < NX; ++i) { mbar_init(fullx + i, 1); mbar_init(xfree + i, 1); }
        for (int i = 0; i < 2; ++i) mbar_init(uready + i, 1);
        for (int i = 0; i < NP; ++i) { mbar_init(phiready + i, kWorkers); mbar_init(pfree + i, 1); }
        for (int i = 0; i < NN; ++i) { mbar_init(numready + i, 1); mbar_init(numfree + i, kWorkers); }
        fence_mbar_init();
    }
    if (warp == 0) { tmem_alloc(tslot, C::TMEM_Q); tmem_relinquish(); }
    stage_phi_table<C>(a, sTe, sAB, sbias, Wop);
    grid_dependency_sync();  // the key statistics and the work split are read from here on
    const Items it(a);
    // padded rows of every item of this block produce zeros (unless the split kernel zeroed them)
    for (int item = it.begin; item < it.end && !a.padded_zeroed; ++item) {
        const ItemRange ir = item_range(a, it, item);
        __nv_bfloat16 *O = static_cast<__nv_bfloat16 *>(a.O) + head_rows(a, ir.bh) * C::DV;
        const int z0 = max(ir.r0, ir.r1);
        for (int e = tid; e < (ir.rend - z0) * C::DV / 8; e += kThreadsTC)
            reinterpret_cast<uint4 *>(O + (size_t)z0 * C::DV)[e] = make_uint4(0, 0, 0, 0);
    }
    fence_proxy_async_smem();
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tbase = *tslot;
    const uint32_t tmem_num = tbase + 2 * C::NU;

    if (warp == kTmaWarp) {
        if (lane == 0) {
            const int T = block_tiles(a, it);
            TileCursor cur;
            cur.start(a, it);
            bool failed = false;
            for (int g = 0; g < T && !failed; ++g, cur.next(a, it)) {
                const int x = g % NX;
                if (g >= NX) wait_or_fail(xfree + x, ((g - NX) / NX) & 1, failed, status);
                mbar_arrive_expect_tx(fullx + x, C::XT);
                for (int kb = 0; kb < C::KBX; ++kb)
                    tma_load_3d(Xb + x * C::XT + kb * 16384, &mapQ, kb * 64, cur.row0(), cur.g.bh, fullx + x);
            }
        }
    } else if (warp == kMmaWarp) {
        if (lane == 0) {
            const int T = block_tiles(a, it);
            const uint64_t dx0 = sdesc(smem_u32(Xb), 16, 1024, kSwizzle128);
            const uint64_t dw0 = sdesc(smem_u32(Wop), 16, 1024, kSwizzle128);
            const uint64_t dp0 = sdesc(smem_u32(Pb), 16, 1024, kSwizzle128);
            const uint64_t ds0 = sdesc(smem_u32(Sop), 16, 1024, kSwizzle128);
            bool failed = false;
            auto proj = [&](int g) {
                const int x = g % NX;
                wait_or_fail(fullx + x, (g / NX) & 1, failed, status);
                tc_fence_after();
                issue_proj<C>(tbase + (g & 1) * C::NU, dadd(dx0, x * C::XT), dw0);
                mma_commit(uready + (g & 1));
                mma_commit(xfree + x);
            };
            if (T > 0) proj(0);
            if (T > 1) proj(1);
            for (int g = 0; g < T && !failed; ++g) {
                const int p = g % NP, q = g % NN;
                wait_or_fail(phiready + p, (g / NP) & 1, failed, status);
                if (g >= NN) wait_or_fail(numfree + q, ((g - NN) / NN) & 1, failed, status);
                tc_fence_after();
                constexpr uint32_t idN = idesc_bf16(128, 2 * C::DV, false, false);
                const uint64_t dp = dadd(dp0, p * C::PT);
#pragma unroll
                for (int kb = 0; kb < C::NPB; ++kb)
#pragma unroll
                    for (int k = 0; k < 4; ++k)
                        mma_bf16_ss(tmem_num + q * 2 * C::DV, dadd(dp, kb * 16384 + 32 * k),
                                    dadd(ds0, kb * (2 * C::DV * 128) + 32 * k), idN, (kb | k) != 0);
                mma_commit(numready + q);
                mma_commit(pfree + p);
                if (g + 2 < T) proj(g + 2);
            }
        }
    } else {
        const int Q = warp >> 2, r = ((warp & 3) << 5) | lane;
        const uint32_t lrow = (uint32_t)((warp & 3) << 5) << 16;
        bool failed = false;
        // O of tile g is written during tile g + 1 (after its feature map and normaliser barrier), so that
        // the numerator product runs while the workers start the next tile
        int pend_g = -1, pend_row = -1;  // tile, and this thread's row of [B*H*n] in it (-1: padded; the
                                         // rows of tensors that fit in device memory stay below 2^31)
        float pend_dsum = 0.0f;
        auto o_out = [&](int gp, int row, float dsum) {
            const int q = gp % NN;
            wait_or_fail(numready + q, (gp / NN) & 1, failed, status);
            tc_fence_after();
            // this thread writes output columns [Q*HC, (Q+1)*HC) of the row
            constexpr int HC = C::DV / 4;
            const float inv = dsum != 0.0f ? 1.0f / dsum : 0.0f;  // one division per row
            uint4 outv[HC / 8];
            const uint32_t col = lrow + tmem_num + q * 2 * C::DV + Q * HC;
            if constexpr (HC == 8) {
                uint32_t xh[8], xl[8];
                tmem_ld8(col, xh);
                tmem_ld8(col + C::DV, xl);
                tmem_wait_ld();
                float o[8];
#pragma unroll
                for (int c = 0; c < 8; ++c) o[c] = (__uint_as_float(xh[c]) + __uint_as_float(xl[c])) * inv;
                outv[0] = make_uint4(pack_bf16x2(o[0], o[1]), pack_bf16x2(o[2], o[3]), pack_bf16x2(o[4], o[5]),
                                     pack_bf16x2(o[6], o[7]));
            } else {
#pragma unroll
                for (int c0 = 0; c0 < HC; c0 += 16) {
                    uint32_t xh[16], xl[16];
                    tmem_ld16(col + c0, xh);
                    tmem_ld16(col + c0 + C::DV, xl);
                    tmem_wait_ld();
                    float o[16];
#pragma unroll
                    for (int c = 0; c < 16; ++c) o[c] = (__uint_as_float(xh[c]) + __uint_as_float(xl[c])) * inv;
#pragma unroll
                    for (int c = 0; c < 16; c += 8)
                        outv[(c0 + c) / 8] =
                            make_uint4(pack_bf16x2(o[c], o[c + 1]), pack_bf16x2(o[c + 2], o[c + 3]),
                                       pack_bf16x2(o[c + 4], o[c + 5]), pack_bf16x2(o[c + 6], o[c + 7]));
                }
            }
            tc_fence_before();
            mbar_arrive(numfree + q);
            if (row >= 0) {
                uint4 *dst = reinterpret_cast<uint4 *>(static_cast<__nv_bfloat16 *>(a.O) + (size_t)row * C::DV + Q * HC);
#pragma unroll
                for (int k = 0; k < HC / 8; ++k) dst[k] = outv[k];
            }
        };
        int g = 0, cur_bh = -1;
        for (int item = it.begin; item < it.end; ++item) {
            const ItemRange ir = item_range(a, it, item);
            if (ir.ntiles == 0) continue;
            if (ir.bh != cur_bh) {
                // operand [S_hi; S_lo]^T and z of this head.  Safe to overwrite once the pending output is
                // written (its contraction, the last to read the operand, is then complete) and every worker
                // has passed the barrier below.
                if (pend_g >= 0) { o_out(pend_g, pend_row, pend_dsum); pend_g = -1; }
                named_sync<kWorkers>(1);
                const float *Sg = a.S_fin + head_state(a, ir.bh) * C::D * C::DV;
                for (int e = tid; e < 2 * C::DV * C::D; e += kWorkers) {
                    const int n = e / C::D, f = e % C::D;
                    __nv_bfloat16 hi, lo;
                    split_bf16(Sg[f * C::DV + (n % C::DV)], hi, lo);
                    *reinterpret_cast<__nv_bfloat16 *>(Sop + (f / 64) * (2 * C::DV * 128) + sw128_chunk(n, (f % 64) / 8) +
                                                       (f % 8) * 2) = (n < C::DV) ? hi : lo;
                }
                for (int e = tid; e < C::D; e += kWorkers) sz[e] = a.z_fin[head_state(a, ir.bh) * C::D + e];
                named_sync<kWorkers>(1);
                cur_bh = ir.bh;
            }
            for (int t = 0; t < ir.ntiles; ++t, ++g) {
                const int p = g % NP;
                const int row0 = ir.r0 + t * 128;
                const int nvalid = min(128, ir.r1 - row0);
                wait_or_fail(uready + (g & 1), (g >> 1) & 1, failed, status);
                if (g >= NP) wait_or_fail(pfree + p, ((g - NP) / NP) & 1, failed, status);
                tc_fence_after();
                const bool valid = r < nvalid;
                float den = 0.0f;
                phi_row_quarter<C>(Q, tbase + lrow + (g & 1) * C::NU, sTe, sAB, sbias, channel_floor(a.lay), valid, r, Pb + p * C::PT, nullptr,
                               nullptr, sz, den);
                float *dslot = sden + (g & 1) * 512;
                dslot[Q * 128 + r] = den;
                fence_proxy_async_smem();
                tc_fence_before();
                mbar_arrive(phiready + p);
                quarter_sync(warp);  // all four parts of this quarter's rows' normalisers are written
                // read now: the slot is written again two tiles on, after the next tile's barrier
                const float dsum = dslot[r] + dslot[128 + r] + dslot[256 + r] + dslot[384 + r] + a.eps;
                if (pend_g >= 0) o_out(pend_g, pend_row, pend_dsum);
                pend_g = g;
                pend_row = valid ? (int)head_rows(a, ir.bh) + row0 + r : -1;
                pend_dsum = dsum;
            }
        }
        if (pend_g >= 0) o_out(pend_g, pend_row, pend_dsum);
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 0) tmem_dealloc(tbase, C::TMEM_Q);
}

// host side

typedef CUresult (*EncodeTiledFn)(CUtensorMap *, CUtensorMapDataType, cuuint32_t, void *, const cuuint64_t *,
                                  const cuuint64_t *, const cuuint32_t *, const cuuint32_t *, CUtensorMapInterleave,
                                  CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn encoder() {
    static EncodeTiledFn fn = nullptr;
    static bool tried = false;
    if (!tried) {
        tried = true;
        void *p = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
                cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<EncodeTiledFn>(p);
    }
    return fn;
}

// (width, n, BH) bf16 tensor, boxes of 64 columns x `rows` rows, 128B swizzle,
// out-of-range elements read as zero.  Head z starts hs_mul * n rows after head z - 1 (hs_mul > 1: one
// head index of each sequence, for per-head parameters).
bool make_map_impl(CUtensorMap *m, const void *base, int width, int n, int BH, int rows = 128, int hs_mul = 1) {
    EncodeTiledFn enc = encoder();
    if (!enc) return false;
    cuuint64_t dims[3] = {(cuuint64_t)width, (cuuint64_t)n, (cuuint64_t)BH};
    cuuint64_t strides[2] = {(cuuint64_t)width * 2, (cuuint64_t)hs_mul * n * width * 2};
    cuuint32_t box[3] = {64, (cuuint32_t)rows, 1};
    cuuint32_t es[3] = {1, 1, 1};
    return enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void *>(base), dims, strides, box, es,
               CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
               CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

int *status_word(const AttnArgs &a) { return reinterpret_cast<int *>(reinterpret_cast<char *>(a.counters) - 256); }

// Work items of the persistent tensor-core kernels: chunks of whole 128-row
// tiles of one head (4 tiles by default; LUNA_TC_TILES_PER_SPLIT overrides it
// for tuning and for tests of long per-item tile loops).  There are never more
// chunks per head than the generic plan sized the partial-sum workspace for.
AttnArgs tc_items_impl(const AttnArgs &a) {
    AttnArgs b = a;
    const int ntile = (a.n + 127) / 128;
    int tiles = 4;
    if (const char *env = getenv("LUNA_TC_TILES_PER_SPLIT")) {
        const int v = atoi(env);
        if (v > 0 && v < (1 << 20)) tiles = v;
    }
    if (tiles > ntile) tiles = ntile > 0 ? ntile : 1;
    while ((ntile + tiles - 1) / tiles > a.nsplit) ++tiles;
    b.rows_per_split = tiles * 128;
    b.nsplit = (ntile + tiles - 1) / tiles;
    return b;
}

// Valid 128-row tiles of work item i (chunk i % nsplit of head i / nsplit).
__device__ __forceinline__ int item_tiles(const AttnArgs &a, int i) {
    const int bh = i / a.nsplit, c = i - bh * a.nsplit;
    const int len = head_length(a.lengths, bh / a.H, a.n);
    const int r0 = c * a.rows_per_split, r1 = min(len, min(a.n, r0 + a.rows_per_split));
    return r1 > r0 ? (r1 - r0 + 127) / 128 : 0;
}

// Split of the work items over a grid of G persistent blocks (one block of 1024 threads): each block gets a
// contiguous, non-empty item range holding about 1/G of the valid tiles (block b starts at the first item
// before which at least b/G of them lie), and each head the first and last block holding one of its items.
// The tile prefix lives in shared memory (kSplitItems items at most; more items keep the split by count).
constexpr int kSplitThreads = 1024;
constexpr int kSplitItems = 12 * 1024;
// Blocks 1.. of the launch zero the rows past each sequence's length of the outputs in zmask (1: O, 2: dQ,
// 4: dK, 8: dV), head by head with the whole GPU's store bandwidth, so that the persistent kernels skip it.
__global__ void __launch_bounds__(kSplitThreads) k_tile_split(AttnArgs a, int G, int zmask) {
    grid_dependency_sync();
    if (blockIdx.x > 0) {
        const int Z = gridDim.x - 1;
        for (int bh = blockIdx.x - 1; bh < a.B * a.H; bh += Z) {
            const int len = head_length(a.lengths, bh / a.H, a.n);
            if (len >= a.n) continue;
            auto zero = [&](void *X, int w) {  // w: bf16 elements per row (a multiple of 8)
                uint4 *p = reinterpret_cast<uint4 *>(static_cast<__nv_bfloat16 *>(X) + (head_rows(a, bh) + len) * w);
                const int cnt = (a.n - len) * (w / 8);
                for (int e = threadIdx.x; e < cnt; e += blockDim.x) p[e] = make_uint4(0, 0, 0, 0);
            };
            if (zmask & 1) zero(a.O, a.dv);
            if (zmask & 2) zero(a.dQ, a.d);
            if (zmask & 4) zero(a.dK, a.d);
            if (zmask & 8) zero(a.dV, a.dv);
        }
        return;
    }
    __shared__ int wsum[kSplitThreads / 32];
    __shared__ int ssplit[kMaxGrid + 1];
    extern __shared__ int prefix[];  // [total + 1] tiles before item i
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int total = a.B * a.H * a.nsplit;
    int *split = a.items_ws;               // [G + 1]
    int *runs = split + kMaxGrid + 1;      // [2 * BH]
    const int per = (total + kSplitThreads - 1) / kSplitThreads;
    const int i0 = min(total, tid * per), i1 = min(total, i0 + per);
    int mine = 0;
    for (int i = i0; i < i1; ++i) {
        const int t = item_tiles(a, i);
        prefix[i] = t;
        mine += t;
    }
    // block-wide scans (warp shuffles, then over the warps); op 0: sum, op 1: max
    auto scan = [&](int v, bool mx) {
        int incl = v;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const int w = __shfl_up_sync(0xffffffffu, incl, o);
            if (lane >= o) incl = mx ? max(incl, w) : incl + w;
        }
        if (lane == 31) wsum[warp] = incl;
        __syncthreads();
        if (warp == 0) {
            int w = wsum[lane];
#pragma unroll
            for (int o = 1; o < 32; o <<= 1) {
                const int u = __shfl_up_sync(0xffffffffu, w, o);
                if (lane >= o) w = mx ? max(w, u) : w + u;
            }
            wsum[lane] = w;
        }
        __syncthreads();
        const int before = warp > 0 ? wsum[warp - 1] : (mx ? INT_MIN : 0);
        const int r = mx ? max(before, incl) : before + incl;  // inclusive over the block
        const int last = wsum[kSplitThreads / 32 - 1];
        __syncthreads();  // wsum is reused by the next scan
        return make_int2(r, last);
    };
    const int2 sc = scan(mine, false);
    int run = sc.x - mine;
    for (int i = i0; i < i1; ++i) {
        const int t = prefix[i];
        prefix[i] = run;
        run += t;
    }
    const int T = sc.y;
    if (tid == 0) prefix[total] = T;
    __syncthreads();
    // lb[b]: first item with at least b*T/G tiles before it.  Every block must get an item (total >= G), so
    // start[b] = b + min(max over b' <= b of (lb[b'] - b'), total - G): strictly increasing, start[0] = 0.
    int lbm = INT_MIN;
    if (tid < G) {
        const long long target = (long long)tid * T / G;
        int lo = 0, hi = total;
        while (lo < hi) {
            const int mid = (lo + hi) >> 1;
            if (prefix[mid] < target) lo = mid + 1; else hi = mid;
        }
        lbm = lo - tid;
    }
    const int2 mx = scan(lbm, true);
    if (tid < G) ssplit[tid] = tid + min(mx.x, total - G);
    if (tid == 0) ssplit[G] = total;
    __syncthreads();
    for (int b = tid; b <= G; b += kSplitThreads) split[b] = ssplit[b];
    // owner of item i: the block b with ssplit[b] <= i < ssplit[b + 1]
    auto owner = [&](int i) {
        int lo = 0, hi = G - 1;
        while (lo < hi) {
            const int mid = (lo + hi + 1) >> 1;
            if (ssplit[mid] <= i) lo = mid; else hi = mid - 1;
        }
        return lo;
    };
    for (int bh = tid; bh < a.B * a.H; bh += kSplitThreads) {
        runs[2 * bh] = owner(bh * a.nsplit);
        runs[2 * bh + 1] = owner((bh + 1) * a.nsplit - 1);
    }
}

// SM count of the current device, cached per device ordinal (host threads may plan for different
// devices at once; a racing first lookup stores the same value twice).
int sm_count_impl() {
    constexpr int kMaxDev = 64;
    static std::atomic<int> cache[kMaxDev];
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return 148;
    if (dev >= 0 && dev < kMaxDev) {
        const int c = cache[dev].load(std::memory_order_relaxed);
        if (c > 0) return c;
    }
    int n = 0;
    if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n <= 0) return 148;
    if (dev >= 0 && dev < kMaxDev) cache[dev].store(n, std::memory_order_relaxed);
    return n;
}

int grid_impl(const AttnArgs &a) {
    const int items = a.B * a.H * a.nsplit;
    return items < sm_count_impl() ? items : sm_count_impl();
}

AttnArgs balanced_impl(const AttnArgs &a0, cudaStream_t s, cudaError_t *err, int zmask) {
    AttnArgs a = tc_items_impl(a0);
    *err = cudaSuccess;
    if (a.split != nullptr || a.lengths == nullptr || a.items_ws == nullptr) return a;
    const int G = grid_impl(a);
    const int total = a.B * a.H * a.nsplit;
    if (G < 1 || G > kMaxGrid || total > kSplitItems) return a;
    const size_t smem = ((size_t)total + 1) * sizeof(int);
    if (smem > 48 * 1024 &&
        (*err = cudaFuncSetAttribute(k_tile_split, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem)) != cudaSuccess)
        return a;
    const int zblocks = zmask ? std::min(a.B * a.H, sm_count_impl()) : 0;
    LUNA_LAUNCH_DEP("tile_split", !a.ch_sigma, k_tile_split, 1 + zblocks, kSplitThreads, smem, s, a, G, zmask);
    if ((*err = cudaGetLastError()) != cudaSuccess) return a;
    a.split = a.items_ws;
    a.runs = a.split + kMaxGrid + 1;
    a.padded_zeroed = zmask != 0;
    return a;
}

template <class C>
cudaError_t keys_tc(const AttnArgs &a, cudaStream_t s) {
    CUtensorMap mK, mV;
    if (!make_map_impl(&mK, a.K, a.d, a.n, a.B * a.H, 128, a.hs_mul) ||
        !make_map_impl(&mV, a.V, a.dv, a.n, a.B * a.H, 128, a.hs_mul))
        return cudaErrorInvalidValue;
    cudaError_t e = cudaFuncSetAttribute(k_tc_keys<C>, cudaFuncAttributeMaxDynamicSharedMemorySize, C::SMEM_K);
    if (e != cudaSuccess) return e;
    LUNA_LAUNCH_DEP("tc_keys", !a.ch_sigma, k_tc_keys<C>, grid_impl(a), kThreadsTC, C::SMEM_K, s, mK, mV, a, status_word(a));
    return cudaGetLastError();
}

template <class C>
cudaError_t fwd_tc(const AttnArgs &a0, cudaStream_t s) {
    cudaError_t e;
    const AttnArgs a = balanced_impl(a0, s, &e, 1);  // the query pass writes O
    if (e != cudaSuccess) return e;
    if ((e = keys_tc<C>(a, s)) != cudaSuccess) return e;
    if ((e = launch_chrms_scale_state(a, s)) != cudaSuccess) return e;
    CUtensorMap mQ;
    if (!make_map_impl(&mQ, a.Q, a.d, a.n, a.B * a.H, 128, a.hs_mul)) return cudaErrorInvalidValue;
    e = cudaFuncSetAttribute(k_tc_query<C>, cudaFuncAttributeMaxDynamicSharedMemorySize, C::SMEM_Q);
    if (e != cudaSuccess) return e;
    LUNA_LAUNCH_DEP("tc_query", !a.ch_sigma, k_tc_query<C>, grid_impl(a), kThreadsTC, C::SMEM_Q, s, mQ, a, status_word(a));
    return cudaGetLastError();
}

using C32 = Cfg<64, 32, 8>;
using C64 = Cfg<64, 64, 8>;
using C128 = Cfg<128, 128, 16>;

int variant(const luna_attn_desc &ad, const TableLayout &lay) {
    if (ad.io != LUNA_BF16 || ad.causal || lay.L != 8 || lay.P > kPpad || ad.d != ad.dv) return -1;
    if (ad.d == 32 && lay.M == 8) return 0;
    if (ad.d == 64 && lay.M == 8) return 1;
    if (ad.d == 128 && lay.M == 16) return 2;
    return -1;
}

}  // namespace

bool tc_make_map(CUtensorMap *m, const void *base, int width, int n, int BH, int hs_mul) {
    return make_map_impl(m, base, width, n, BH, 128, hs_mul);
}
bool tc_make_map_rows(CUtensorMap *m, const void *base, int width, int n, int BH, int rows, int hs_mul) {
    return make_map_impl(m, base, width, n, BH, rows, hs_mul);
}
int tc_sm_count() { return sm_count_impl(); }
AttnArgs tc_work_items(const AttnArgs &a) { return tc_items_impl(a); }
AttnArgs tc_balanced_items(const AttnArgs &a, cudaStream_t s, cudaError_t *err, int zmask) {
    return balanced_impl(a, s, err, zmask);
}
int tc_grid(const AttnArgs &items) { return grid_impl(items); }

TcPlan tc_plan(const luna_attn_desc &ad, const TableLayout &lay) {
    TcPlan p;
    if (lay_variant(lay)) return p;  // the feature-map variants run on the generic kernels
    p.variant = variant(ad, lay);
    p.eligible = p.variant >= 0 && encoder() != nullptr;
    p.bwd = p.eligible && tc_bwd_supported(ad, lay);
    if (ad.causal) {
        luna_attn_desc nc = ad;
        nc.causal = 0;
        p.causal_fwd = encoder() != nullptr && variant(nc, lay) >= 0 && tc_causal_supported(ad, lay);
        p.causal_bwd = p.causal_fwd;
    }
    return p;
}

bool tc_inputs_ok(const TcPlan &p, const void *a, const void *b, const void *c, const void *d) {
    auto al = [](const void *x) { return x == nullptr || (reinterpret_cast<uintptr_t>(x) & 15) == 0; };
    return p.eligible && al(a) && al(b) && al(c) && al(d);
}

cudaError_t launch_tc_fwd(const TcPlan &p, const AttnArgs &a, char *, cudaStream_t s) {
    switch (p.variant) {
        case 0: return fwd_tc<C32>(a, s);
        case 1: return fwd_tc<C64>(a, s);
        case 2: return fwd_tc<C128>(a, s);
    }
    return cudaErrorNotSupported;
}

cudaError_t launch_tc_keys_items(const AttnArgs &a, cudaStream_t s) {
    const TcPlan p = tc_plan(luna_attn_desc{a.B, a.H, a.n, a.d, a.dv, 0, 0, a.eps, LUNA_BF16}, a.lay);
    switch (p.variant) {
        case 0: return keys_tc<C32>(a, s);
        case 1: return keys_tc<C64>(a, s);
        case 2: return keys_tc<C128>(a, s);
    }
    return cudaErrorNotSupported;
}

cudaError_t launch_tc_stats(const AttnArgs &a0, cudaStream_t s) {
    const TcPlan p = tc_plan(luna_attn_desc{a0.B, a0.H, a0.n, a0.d, a0.dv, 0, 0, a0.eps, LUNA_BF16}, a0.lay);
    cudaError_t e;
    const AttnArgs a = balanced_impl(a0, s, &e, 0);  // the split of the forward pass: the same sums in the same order
    if (e != cudaSuccess) return e;
    switch (p.variant) {
        case 0: e = keys_tc<C32>(a, s); break;
        case 1: e = keys_tc<C64>(a, s); break;
        case 2: e = keys_tc<C128>(a, s); break;
        default: return cudaErrorNotSupported;
    }
    if (e != cudaSuccess) return e;
    return launch_chrms_scale_state(a, s);
}

cudaError_t launch_tc_bwd(const TcPlan &p, const AttnArgs &a, char *, bool have_stats, cudaStream_t s) {
    if (p.bwd && tc_bwd_fits(a)) return launch_tc_bwd_kernels(a, have_stats, s);
    if (!have_stats) {  // generic backward on the statistics of the tensor-core key pass
        cudaError_t e = launch_tc_stats(a, s);
        if (e != cudaSuccess) return e;
    }
    return launch_simt_bwd(a, LUNA_BF16, true, s);
}

}  // namespace luna
