// Chain rule through the feature map on tensor cores (bf16 I/O, d = 128,
// M = 16 projections, L = 8 channels), for a gradient dphi that an earlier
// kernel left in global memory (fp32, one row of D = 128 features per token).
//
// Per 128-row tile of X (Q or K):
//   MMA   U = X [W_hi; W_mid; W_lo; 0]^T        (u as accurate as fp32: it decides the kinks)
//   work  interval search, alpha of the 8 channels, g = dphi on active outputs,
//         dU = sum_l g alpha, histogram of (g, g u); tile G = [dU_hi | dU_lo | dU_hi | 0]
//   MMA   dX = G [W_hi; W_hi; W_lo; 0],  dW^T += X^T [dU_hi | dU_lo]
// The block's parameter-gradient partial (dW, db, histogram) goes to its slot
// of the partial buffer; the common reduction kernels finish them.
#include "luna_tc_bwd_dev.cuh"

namespace luna {
namespace {
using namespace sm100;
using namespace simt;
using namespace tcdev;
using namespace tcbwd;

struct P128 {
    static constexpr int d = 128, DX = 128, MP = 16, D = 128, NU = 64, PP = MP / kBRowThreads;
    static constexpr int KBX = DX / 64;
    static constexpr uint32_t TILE = 16384;      // 128 rows x 128 B
    static constexpr uint32_t XT = KBX * TILE;   // X tile
    static constexpr uint32_t WOP = KBX * NU * 128;
    static constexpr uint32_t WX = d * 128;      // dX operand: output-column rows, K = 64
    static constexpr int NS = 2;
    static constexpr uint32_t SMEM = NS * XT + TILE + WOP + WX + kTableBytes + kNint * 16 * 4 + MP * d * 4 + 64 +
                                     2 * (kBWorkers / 32) * 4 + kBarBytes + 1024;
    static_assert(SMEM <= kSmemLimit, "shared memory budget");
    static_assert(PP == 4, "four projections per thread");
    static_assert(hist_tiles<MP>() == 8, "eight 2048-sample tiles per histogram group");
};

// [W_hi; W_hi; W_lo; 0] (16 rows each) as the K-major B operand of dX = G W: row n = output column.
template <class C>
__device__ void stage_wx64(const AttnArgs &a, uint8_t *dst) {
    const float *W = reinterpret_cast<const float *>(a.table + a.lay.off_W);
    for (int e = threadIdx.x; e < C::d * 64; e += blockDim.x) {
        const int n = e / 64, k = e % 64, part = k / C::MP;
        float v = 0.0f;
        if (part < 3) {
            __nv_bfloat16 hi, lo;
            split_bf16(W[(k % C::MP) * a.d + n], hi, lo);
            v = part < 2 ? __bfloat162float(hi) : __bfloat162float(lo);
        }
        *reinterpret_cast<__nv_bfloat16 *>(dst + sw128_chunk(n, k / 8) + (k % 8) * 2) = __float2bfloat16_rn(v);
    }
}

template <class C>
__global__ void __launch_bounds__(kBThreads, 1)
    k_tc_phi_bwd(const __grid_constant__ CUtensorMap mapX, AttnArgs a, const float *dphi, __nv_bfloat16 *dXg,
                 int slot0, const float *kfold, int *status) {
    extern __shared__ uint8_t smem_raw[];
    const float fl = channel_floor(a.lay);  // lower bound of a channel output
    uint8_t *sm = align1024(smem_raw);
    constexpr int NS = C::NS;
    constexpr uint32_t T16 = C::TILE;
    uint8_t *Xb = sm;                     // [NS] X tiles
    uint8_t *Gt = Xb + NS * C::XT;        // G = [dU_hi | dU_lo | dU_hi | 0]
    uint8_t *Wop = Gt + T16;
    uint8_t *Wx = Wop + C::WOP;
    float *sTe = reinterpret_cast<float *>(Wx + C::WX);
    float *sAB = sTe + kEytzinger;
    float *sbias = sAB + kNint * 16;
    int *bins = reinterpret_cast<int *>(sbias + 32);
    float *sdW = reinterpret_cast<float *>(bins + kNint * 16);  // [M][d]
    float *sdb = sdW + C::MP * C::d;                            // [M]
    float *smax = sdb + 16;
    uint64_t *bars = reinterpret_cast<uint64_t *>(smax + 2 * (kBWorkers / 32));
    uint64_t *fullx = bars;              // [NS]
    uint64_t *xfree = fullx + NS;        // [NS] projection and dW^T consumed the X tile
    uint64_t *uready = xfree + NS;       // [2]
    uint64_t *gready = uready + 2;       // [1] count 512
    uint64_t *gfree = gready + 1;        // [1]
    uint64_t *dxready = gfree + 1;       // [1]
    uint64_t *dxfree = dxready + 1;      // [1] count 512
    uint64_t *wdone = dxfree + 1;        // [1]
    uint32_t *tslot = reinterpret_cast<uint32_t *>(wdone + 1);
    static_assert((2 * NS + 7) * 8 + 4 <= kBarBytes, "barrier area");

    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const Items it(a);
    // TMEM: U [2 x 64] | dX [128] | dW^T [32]
    constexpr uint32_t cU = 0, cX = 128, cW = 256;
    const int slot = slot0 + (int)blockIdx.x;

    if (tid == 0) {
        for (int i = 0; i < NS; ++i) { mbar_init(fullx + i, 1); mbar_init(xfree + i, 1); }
        for (int i = 0; i < 2; ++i) mbar_init(uready + i, 1);
        mbar_init(gready, kBWorkers); mbar_init(gfree, 1);
        mbar_init(dxready, 1); mbar_init(dxfree, kBWorkers);
        mbar_init(wdone, 1);
        fence_mbar_init();
    }
    if (warp == 0) { tmem_alloc(tslot, 512); tmem_relinquish(); }
    stage_phi_table<C>(a, sTe, sAB, sbias, Wop);
    stage_wx64<C>(a, Wx);
    for (int e = tid; e < kNint * 16; e += blockDim.x) bins[e] = 0;
    for (int e = tid; e < C::MP * C::d + 16; e += blockDim.x) sdW[e] = 0.0f;
    for (int e = tid; e < (int)(T16 / 16); e += blockDim.x) reinterpret_cast<uint4 *>(Gt)[e] = make_uint4(0, 0, 0, 0);
    float *hpart = a.gpart + (size_t)slot * a.gsize + C::MP * a.d + C::MP;
    for (int e = tid; e < a.lay.nint * 16; e += blockDim.x) hpart[e] = 0.0f;
    for (int item = it.begin; item < it.end; ++item) {  // padded rows receive zero gradients
        const ItemRange ir = item_range(a, it, item);
        __nv_bfloat16 *dX = dXg + head_rows(a, ir.bh) * C::d;
        const int z0 = max(ir.r0, ir.r1);
        for (int e = tid; e < (ir.rend - z0) * C::d / 8; e += blockDim.x)
            reinterpret_cast<uint4 *>(dX + (size_t)z0 * C::d)[e] = make_uint4(0, 0, 0, 0);
    }
    fence_proxy_async_smem();
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tbase = *tslot;
    const int T = block_tiles(a, it);

    if (warp == kBTma) {
        if (lane == 0) {
            TileCursor cur;
            cur.start(a, it);
            bool failed = false;
            for (int g = 0; g < T && !failed; ++g, cur.next(a, it)) {
                const int s = g % NS;
                if (g >= NS) wait_or_fail(xfree + s, ((g - NS) / NS) & 1, failed, status);
                mbar_arrive_expect_tx(fullx + s, C::XT);
                for (int kb = 0; kb < C::KBX; ++kb)
                    tma_load_3d(Xb + s * C::XT + kb * T16, &mapX, kb * 64, cur.row0(), cur.g.bh, fullx + s);
            }
        }
    } else if (warp == kBMma) {
        if (lane == 0) {
            const uint64_t dXk = sdesc(smem_u32(Xb), 16, 1024, kSwizzle128);      // K-major (rows = tokens)
            const uint64_t dXm = sdesc(smem_u32(Xb), T16, 1024, kSwizzle128);     // MN-major (M = input columns)
            const uint64_t dWo = sdesc(smem_u32(Wop), 16, 1024, kSwizzle128);
            const uint64_t dWx = sdesc(smem_u32(Wx), 16, 1024, kSwizzle128);
            const uint64_t dGk = sdesc(smem_u32(Gt), 16, 1024, kSwizzle128);      // K-major A of dX
            const uint64_t dGm = sdesc(smem_u32(Gt), T16, 1024, kSwizzle128);     // MN-major B of dW^T
            bool failed = false;
            auto proj = [&](int g) {
                const int s = g % NS;
                wait_or_fail(fullx + s, (g / NS) & 1, failed, status);
                tc_fence_after();
                constexpr uint32_t idU = idesc_bf16(128, C::NU, false, false);
#pragma unroll
                for (int kb = 0; kb < C::KBX; ++kb)
#pragma unroll
                    for (int k = 0; k < 4; ++k)
                        mma_bf16_ss(tbase + cU + (g & 1) * C::NU, dadd(dXk, s * C::XT + kb * T16 + 32 * k),
                                    dadd(dWo, kb * (C::NU * 128) + 32 * k), idU, (kb | k) != 0);
                mma_commit(uready + (g & 1));
            };
            if (T > 0) proj(0);
            if (T > 1) proj(1);
            for (int g = 0; g < T && !failed; ++g) {
                const int s = g % NS;
                // dX = G [W_hi; W_hi; W_lo; 0] and dW^T += X^T [dU_hi | dU_lo]
                wait_or_fail(gready, g & 1, failed, status);
                if (g >= 1) wait_or_fail(dxfree, (g - 1) & 1, failed, status);
                tc_fence_after();
                constexpr uint32_t idX = idesc_bf16(128, C::d, false, false);
#pragma unroll
                for (int k = 0; k < 4; ++k) mma_bf16_ss(tbase + cX, dadd(dGk, 32 * k), dadd(dWx, 32 * k), idX, k != 0);
                mma_commit(dxready);  // before the dW^T products: the workers wait for dX only
                constexpr uint32_t idW = idesc_bf16(128, 2 * C::MP, true, true);
#pragma unroll
                for (int k = 0; k < 8; ++k)
                    mma_bf16_ss(tbase + cW, dadd(dXm, s * C::XT + 2048 * k), dadd(dGm, 2048 * k), idW,
                                (g > 0 || k > 0) ? 1u : 0u);
                mma_commit(gfree);
                mma_commit(xfree + s);
                if (g + 2 < T) proj(g + 2);  // the workers read U(g) before gready
            }
            if (T > 0 && !failed) mma_commit(wdone);
            else mbar_arrive(wdone);
        }
    } else {
        // workers: thread (H, r) owns row r of the tile and projections H*PP .. H*PP+PP-1
        const int H = warp >> 2, r = ((warp & 3) << 5) | lane;
        const uint32_t lrow = (uint32_t)((warp & 3) << 5) << 16;
        bool failed = false;
        float db_acc[C::PP];
#pragma unroll
        for (int q = 0; q < C::PP; ++q) db_acc[q] = 0.0f;
        float kf[8];  // channel normalisation: dphi += M kappa_l phi (the scale term, on the scaled table)
#pragma unroll
        for (int l = 0; l < 8; ++l) kf[l] = kfold ? (float)C::MP * kfold[l] : 0.0f;
        HistAcc hacc;
        int g = 0;
        for (int item = it.begin; item < it.end; ++item) {
            const ItemRange ir = item_range(a, it, item);
            __nv_bfloat16 *dX = dXg + head_rows(a, ir.bh) * C::d;
            for (int t = 0; t < ir.ntiles; ++t, ++g) {
                const int row0 = ir.r0 + t * 128;
                const bool valid = r < min(128, ir.r1 - row0);
                const float *dp = dphi + ((size_t)ir.bh * a.n + row0 + r) * C::D + H * C::PP * 8;
                // this thread's 32 dphi values, requested before the waits and the search: one 32-byte
                // load per projection (a whole sector; dphi rows are 512 bytes, 32-byte aligned)
                float4 pv[C::PP][2];
#pragma unroll
                for (int q = 0; q < C::PP; ++q) {
                    pv[q][0] = pv[q][1] = make_float4(0.f, 0.f, 0.f, 0.f);
                    if (valid) ld_cg_v8(dp + 8 * q, pv[q][0], pv[q][1]);
                }
                wait_or_fail(uready + (g & 1), (g >> 1) & 1, failed, status);
                tc_fence_after();
                float u[C::PP];
                int j[C::PP];
                {
                    uint32_t xh[4], xm[4], xl[4];
                    const uint32_t ucol = tbase + lrow + cU + (g & 1) * C::NU + H * C::PP;
                    tmem_ld4(ucol, xh);
                    tmem_ld4(ucol + C::MP, xm);
                    tmem_ld4(ucol + 2 * C::MP, xl);
                    tmem_wait_ld();
#pragma unroll
                    for (int q = 0; q < C::PP; ++q)
                        u[q] = (__uint_as_float(xh[q]) + __uint_as_float(xm[q])) + __uint_as_float(xl[q]) +
                               sbias[H * C::PP + q];
                }
                search<C::PP>(sTe, u, j);
                bool hon = hacc.open;
                float dU[C::PP], gv[C::PP][8];
#pragma unroll
                for (int q = 0; q < C::PP; ++q) {
                    float al[8], y[8];
                    channel_eval(sAB, j[q], u[q], fl, al, y);
                    const float4 p0 = pv[q][0], p1 = pv[q][1];
                    const float dv[8] = {p0.x, p0.y, p0.z, p0.w, p1.x, p1.y, p1.z, p1.w};
                    float du = 0.0f;
#pragma unroll
                    for (int l = 0; l < 8; ++l) {
                        const float gl = (valid && y[l] > fl) ? fmaf(kf[l], y[l], dv[l]) : 0.0f;
                        gv[q][l] = gl;
                        du = fmaf(gl, al[l], du);
                    }
                    dU[q] = du;
                    db_acc[q] += du;
                }
                if (g >= 1) wait_or_fail(gfree, (g - 1) & 1, failed, status);
                {
                    uint32_t h0, l0, h1, l1;
                    const float d01[2] = {dU[0], dU[1]}, d23[2] = {dU[2], dU[3]};
                    dU_pack(d01, h0, l0);
                    dU_pack(d23, h1, l1);
                    const uint32_t off = (H & 1) * 8;
                    *reinterpret_cast<uint2 *>(Gt + sw128_chunk(r, H >> 1) + off) = make_uint2(h0, h1);
                    *reinterpret_cast<uint2 *>(Gt + sw128_chunk(r, 2 + (H >> 1)) + off) = make_uint2(l0, l1);
                    *reinterpret_cast<uint2 *>(Gt + sw128_chunk(r, 4 + (H >> 1)) + off) = make_uint2(h0, h1);
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
                // dX
                wait_or_fail(dxready, g & 1, failed, status);
                tc_fence_after();
                {
                    uint32_t x0[16], x1[16];
                    tmem_ld16(tbase + lrow + cX + 32 * H, x0);
                    tmem_ld16(tbase + lrow + cX + 32 * H + 16, x1);
                    tmem_wait_ld();
                    tc_fence_before();
                    mbar_arrive(dxfree);
                    if (valid) {
                        uint4 *dst = reinterpret_cast<uint4 *>(dX + (size_t)(row0 + r) * C::d + 32 * H);
#pragma unroll
                        for (int k = 0; k < 2; ++k) {
                            float f0[8], f1[8];
#pragma unroll
                            for (int c = 0; c < 8; ++c) {
                                f0[c] = __uint_as_float(x0[8 * k + c]);
                                f1[c] = __uint_as_float(x1[8 * k + c]);
                            }
                            dst[k] = pack8(f0);
                            dst[2 + k] = pack8(f1);
                        }
                    }
                }
            }
        }
        if (hacc.tiles > 0) hist_close(bins, hpart, a.lay.nint, hacc, tid, false, smax, warp, lane);
#pragma unroll
        for (int q = 0; q < C::PP; ++q) {
            float v = db_acc[q];
#pragma unroll
            for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
            if (lane == 0) atomicAdd(sdb + H * C::PP + q, v);
        }
        if (warp < 4) {  // dW^T accumulator: lane = input column, columns [dU_hi | dU_lo] of the projections
            if (T > 0) wait_or_fail(wdone, 0, failed, status);
            tc_fence_after();
            uint32_t x0[16], x1[16];
            tmem_ld16(tbase + ((uint32_t)(warp << 5) << 16) + cW, x0);
            tmem_ld16(tbase + ((uint32_t)(warp << 5) << 16) + cW + 16, x1);
            tmem_wait_ld();
            const int cd = (warp << 5) | lane;
            if (T > 0)
#pragma unroll
                for (int i = 0; i < C::MP; ++i) sdW[i * C::d + cd] = __uint_as_float(x0[i]) + __uint_as_float(x1[i]);
        }
    }
    tc_fence_before();
    __syncthreads();
    store_param_partial<C>(a, sdW, sdb, a.gpart + (size_t)slot * a.gsize);
    __syncthreads();
    if (warp == 0) tmem_dealloc(tbase, 512);
}

}  // namespace

bool tc_make_map(CUtensorMap *m, const void *base, int width, int n, int BH, int hs_mul);
int tc_sm_count();

// Chain rule through the feature map for X in {Q, K}: dphi (fp32, [BH][n][D]) -> dX
// and the parameter-gradient partials of blocks slot0 .. slot0 + grid - 1.
// Work items: a.rows_per_split rows (whole 128-row tiles) of one head.
cudaError_t launch_tc_phi_bwd(const AttnArgs &a, const void *X, const float *dphi, void *dX, int slot0, int grid,
                              cudaStream_t s, const float *kfold) {
    using C = P128;
    CUtensorMap mX;
    if (!tc_make_map(&mX, X, a.d, a.n, a.B * a.H, a.hs_mul)) return cudaErrorInvalidValue;
    cudaError_t e = cudaFuncSetAttribute(k_tc_phi_bwd<C>, cudaFuncAttributeMaxDynamicSharedMemorySize, C::SMEM);
    if (e != cudaSuccess) return e;
    int *st = reinterpret_cast<int *>(reinterpret_cast<char *>(a.counters) - 256);
    LUNA_LAUNCH("tc_phi_bwd", k_tc_phi_bwd<C>, grid, kBThreads, C::SMEM, s, mX, a, dphi,
                static_cast<__nv_bfloat16 *>(dX), slot0, kfold, st);
    return cudaGetLastError();
}

}  // namespace luna
