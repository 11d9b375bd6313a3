// The scale term of the channel RMS normalisation on tensor cores (non-causal
// form, bf16, d = 32 or 64, M = 8, L = 8): with s_l depending on every sample of
// its channel, the gradient reaching the MLP output of each sample of one side
// gains M kappa_l phi_l (kappa from the statistics and the main backward pass).
// This pass adds that term's chain rule to dQ (blockIdx.y = 0) or dK (1) and
// writes its parameter-gradient partials after the main ones, at
// gpart[(side * gridDim.x + blockIdx.x) * gsize].
//
// Per 128-row tile (warp roles as in the backward kernels):
//   TMA   X tile into one of three stages
//   MMA   U = X [W_hi; W_mid; W_lo; 0]^T into one of two TMEM buffers
//   work  u, interval, phi of the 8 channels, g_l = M kappa_l phi_l on active outputs,
//         dU = sum_l g_l alpha_l, the fixed-point interval histogram; tile G = [dU_hi | dU_lo | dU_hi | 0]
//   MMA   dX = G [W_hi; W_hi; W_lo; 0],  dW^T += X^T [dU_hi | dU_lo]
//   work  dX added to the rows of dQ or dK
// The tiles of a side are dealt to the blocks round robin; every role walks the same sequence.
#include "luna_tc_bwd_dev.cuh"

namespace luna {

bool tc_make_map(CUtensorMap *m, const void *base, int width, int n, int BH, int hs_mul);
int tc_sm_count();

namespace {
using namespace sm100;
using namespace simt;
using namespace tcdev;
using namespace tcbwd;

template <int D_>
struct KCfg {
    static constexpr int d = D_, DX = 64, MP = 8, NU = 32, PP = MP / kBRowThreads, NKD = d / 16;
    static constexpr uint32_t TILE = 16384;  // 128 rows x 128 B
    static constexpr int NX = 3;
    static constexpr uint32_t WOP = NU * 128;  // projection operand: NU rows x 64 columns
    static constexpr uint32_t WX = d * 128;    // dX operand: a row per output column, K = 32
    static constexpr uint32_t SMEM = NX * TILE + TILE + WOP + WX + kTableBytes + kNint * 16 * 4 + MP * d * 4 + 64 +
                                     2 * (kBWorkers / 32) * 4 + 64 + kBarBytes + 1024;
    static_assert(SMEM <= kSmemLimit, "shared memory budget");
    static_assert(PP == 2, "two projections per thread");
};

__device__ __forceinline__ bool kterm_tile(const AttnArgs &a, int64_t t, int nt, int &row0, int &bh) {
    bh = (int)(t / nt);
    row0 = (int)(t - (int64_t)bh * nt) * 128;
    return row0 < head_length(a.lengths, bh / a.H, a.n);
}

template <class C>
__global__ void __launch_bounds__(kBThreads, 1)
    k_tc_kterm(const __grid_constant__ CUtensorMap mapQ, const __grid_constant__ CUtensorMap mapK, AttnArgs a,
               const float *kappa, float *gpart, int *status) {
    extern __shared__ uint8_t smem_raw[];
    uint8_t *sm = align1024(smem_raw);
    constexpr int NX = C::NX, PP = C::PP;
    constexpr uint32_t T16 = C::TILE;
    uint8_t *Xb = sm;                 // [NX] X tiles
    uint8_t *Gt = Xb + NX * T16;      // G = [dU_hi | dU_lo | dU_hi | 0]
    uint8_t *Wop = Gt + T16;
    uint8_t *Wx = Wop + C::WOP;
    float *sTe = reinterpret_cast<float *>(Wx + C::WX);
    float *sAB = sTe + kEytzinger;
    float *sbias = sAB + kNint * 16;
    int *bins = reinterpret_cast<int *>(sbias + 32);
    float *sdW = reinterpret_cast<float *>(bins + kNint * 16);  // [M][d]
    float *sdb = sdW + C::MP * C::d;                            // [M] (padded to 16)
    float *smax = sdb + 16;                                     // [2][worker warps]
    float *sk = smax + 2 * (kBWorkers / 32);                    // [8] M kappa_l of this side
    uint64_t *bars = reinterpret_cast<uint64_t *>(sk + 16);
    uint64_t *fullx = bars;            // [NX]
    uint64_t *xfree = fullx + NX;      // [NX] projection and dW^T consumed the X tile
    uint64_t *uready = xfree + NX;     // [2]
    uint64_t *ufree = uready + 2;      // [2] count 512
    uint64_t *gready = ufree + 2;      // [1] count 512
    uint64_t *gfree = gready + 1;      // [1]
    uint64_t *dxready = gfree + 1;     // [1]
    uint64_t *dxfree = dxready + 1;    // [1] count 512
    uint64_t *wdone = dxfree + 1;      // [1]
    uint32_t *tslot = reinterpret_cast<uint32_t *>(wdone + 1);
    static_assert((2 * NX + 9) * 8 + 4 <= kBarBytes, "barrier area");

    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int side = blockIdx.y;
    const int nt = (a.n + 127) / 128;
    const int64_t tiles = (int64_t)a.B * a.H * nt;
    float *gp = gpart + ((size_t)side * gridDim.x + blockIdx.x) * a.gsize;
    float *hpart = gp + C::MP * a.d + C::MP;  // histogram part of the partial
    // TMEM: U [2 x 32] | dX [64] | dW^T (M = 64) [16]
    constexpr uint32_t cU = 0, cX = 64, cW = 128;

    if (tid == 0) {
        for (int i = 0; i < NX; ++i) { mbar_init(fullx + i, 1); mbar_init(xfree + i, 1); }
        for (int i = 0; i < 2; ++i) { mbar_init(uready + i, 1); mbar_init(ufree + i, kBWorkers); }
        mbar_init(gready, kBWorkers); mbar_init(gfree, 1);
        mbar_init(dxready, 1); mbar_init(dxfree, kBWorkers);
        mbar_init(wdone, 1);
        fence_mbar_init();
    }
    if (warp == 0) { tmem_alloc(tslot, 256); tmem_relinquish(); }
    stage_phi_table<C>(a, sTe, sAB, sbias, Wop);
    stage_wx<C>(a, Wx, 0);
    for (int e = tid; e < kNint * 16; e += blockDim.x) bins[e] = 0;
    for (int e = tid; e < C::MP * C::d + 16; e += blockDim.x) sdW[e] = 0.0f;
    for (int e = tid; e < (int)(T16 / 16); e += blockDim.x) reinterpret_cast<uint4 *>(Gt)[e] = make_uint4(0, 0, 0, 0);
    for (int e = tid; e < a.lay.nint * 16; e += blockDim.x) hpart[e] = 0.0f;
    if (tid < 8) sk[tid] = kappa[side * kMaxL + tid] * (float)C::MP;
    fence_proxy_async_smem();
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tbase = *tslot;

    if (warp == kBTma) {
        if (lane == 0) {
            const CUtensorMap *map = side ? &mapK : &mapQ;
            bool failed = false;
            int g = 0, row0, bh;
            for (int64_t t = blockIdx.x; t < tiles && !failed; t += gridDim.x) {
                if (!kterm_tile(a, t, nt, row0, bh)) continue;
                const int x = g % NX;
                if (g >= NX) wait_or_fail(xfree + x, ((g - NX) / NX) & 1, failed, status);
                mbar_arrive_expect_tx(fullx + x, T16);
                tma_load_3d(Xb + x * T16, map, 0, row0, bh, fullx + x);
                ++g;
            }
        }
    } else if (warp == kBMma) {
        if (lane == 0) {
            const uint64_t dXk = sdesc(smem_u32(Xb), 16384, 1024, kSwizzle128);  // K-major (rows = tokens)
            const uint64_t dWo = sdesc(smem_u32(Wop), 16, 1024, kSwizzle128);
            const uint64_t dWx = sdesc(smem_u32(Wx), 16, 1024, kSwizzle128);
            const uint64_t dG = sdesc(smem_u32(Gt), 16384, 1024, kSwizzle128);
            bool failed = false;
            int T = 0, row0, bh;
            for (int64_t t = blockIdx.x; t < tiles; t += gridDim.x) T += kterm_tile(a, t, nt, row0, bh) ? 1 : 0;
            auto proj = [&](int g) {
                const int x = g % NX, b = g & 1;
                wait_or_fail(fullx + x, (g / NX) & 1, failed, status);
                if (g >= 2) wait_or_fail(ufree + b, ((g - 2) >> 1) & 1, failed, status);
                tc_fence_after();
                constexpr uint32_t idU = idesc_bf16(128, C::NU, false, false);
#pragma unroll
                for (int k = 0; k < C::NKD; ++k)
                    mma_bf16_ss(tbase + cU + b * C::NU, dadd(dXk, x * T16 + 32 * k), dadd(dWo, 32 * k), idU, k != 0);
                mma_commit(uready + b);
            };
            if (T > 0) proj(0);
            if (T > 1) proj(1);
            for (int g = 0; g < T && !failed; ++g) {
                const int x = g % NX;
                wait_or_fail(gready, g & 1, failed, status);
                if (g >= 1) wait_or_fail(dxfree, (g - 1) & 1, failed, status);
                tc_fence_after();
                // dX = [dU_hi | dU_lo | dU_hi | 0] [W_hi; W_hi; W_lo; 0], its barrier committed at once
                constexpr uint32_t idX = idesc_bf16(128, C::d, false, false);
#pragma unroll
                for (int k = 0; k < 2; ++k) mma_bf16_ss(tbase + cX, dadd(dG, 32 * k), dadd(dWx, 32 * k), idX, k != 0);
                mma_commit(dxready);
                // dW^T += X^T [dU_hi | dU_lo]: rows = input columns
                constexpr uint32_t idW = idesc_bf16(64, 16, true, true);
#pragma unroll
                for (int k = 0; k < 8; ++k)
                    mma_bf16_ss(tbase + cW, dadd(dXk, x * T16 + 2048 * k), dadd(dG, 2048 * k), idW,
                                (g > 0 || k > 0) ? 1u : 0u);
                mma_commit(gfree);
                mma_commit(xfree + x);
                if (g + 2 < T) proj(g + 2);
            }
            if (T > 0 && !failed) mma_commit(wdone);
            else mbar_arrive(wdone);
        }
    } else {
        // workers: thread (H, r) owns row r of the tile and projections H*PP .. H*PP+PP-1
        const int H = warp >> 2, r = ((warp & 3) << 5) | lane;
        const uint32_t lrow = (uint32_t)((warp & 3) << 5) << 16;
        __nv_bfloat16 *dXg = static_cast<__nv_bfloat16 *>(side ? a.dK : a.dQ);
        bool failed = false;
        float db_acc[PP] = {};
        HistAcc hacc;
        int g = 0, row0, bh;
        for (int64_t t = blockIdx.x; t < tiles; t += gridDim.x) {
            if (!kterm_tile(a, t, nt, row0, bh)) continue;
            const bool valid = row0 + r < head_length(a.lengths, bh / a.H, a.n);
            const int b = g & 1;
            wait_or_fail(uready + b, (g >> 1) & 1, failed, status);
            tc_fence_after();
            float u[PP];
            int j[PP];
            {
                uint32_t xh[2], xm[2], xl[2];
                const uint32_t ucol = tbase + lrow + cU + b * C::NU + H * PP;
                tmem_ld2(ucol, xh);
                tmem_ld2(ucol + C::MP, xm);
                tmem_ld2(ucol + 2 * C::MP, xl);
                tmem_wait_ld();
#pragma unroll
                for (int q = 0; q < PP; ++q)
                    u[q] = (__uint_as_float(xh[q]) + __uint_as_float(xm[q])) + __uint_as_float(xl[q]) +
                           sbias[H * PP + q];
            }
            tc_fence_before();
            mbar_arrive(ufree + b);  // U(g) read: the buffer takes the projection two tiles on
            search<PP>(sTe, u, j);
            float dU[PP], gv[PP][8];
#pragma unroll
            for (int q = 0; q < PP; ++q) {
                float al[8], y[8];
                channel_eval(sAB, j[q], u[q], 0.0f, al, y);
                float du = 0.0f;
#pragma unroll
                for (int l = 0; l < 8; ++l) {
                    const float gl = (valid && y[l] > 0.0f) ? sk[l] * y[l] : 0.0f;  // through the outer ReLU
                    gv[q][l] = gl;
                    du = fmaf(gl, al[l], du);
                }
                dU[q] = du;
                db_acc[q] += du;
            }
            if (g >= 1) wait_or_fail(gfree, (g - 1) & 1, failed, status);
            {  // columns 0 + PP*H: dU_hi;  8 + PP*H: dU_lo;  16 + PP*H: dU_hi (chunks 0, 1, 2)
                uint32_t vh, vl;
                dU_pack(dU, vh, vl);
                *reinterpret_cast<uint32_t *>(Gt + sw128_chunk(r, 0) + H * 4) = vh;
                *reinterpret_cast<uint32_t *>(Gt + sw128_chunk(r, 1) + H * 4) = vl;
                *reinterpret_cast<uint32_t *>(Gt + sw128_chunk(r, 2) + H * 4) = vh;
            }
            fence_proxy_async_smem();
            tc_fence_before();
            mbar_arrive(gready);
            bool hon = hacc.open;
            if (!hon) {  // first tile with a nonzero g in the block: its maxima give the first scales
                float m0 = 0.0f, m1 = 0.0f;
#pragma unroll
                for (int q = 0; q < PP; ++q)
#pragma unroll
                    for (int l = 0; l < 8; ++l) {
                        m0 = finite_max(m0, gv[q][l]);
                        m1 = finite_max(m1, gv[q][l] * u[q]);
                    }
                hon = hist_open(hacc, m0, m1, smax, warp, lane);
            }
            if (hon) {
                hist_add<PP>(bins, hpart, hacc, j, u, gv, dU);
                if (++hacc.tiles == hist_tiles<C::MP>()) hist_close(bins, hpart, a.lay.nint, hacc, tid, true, smax, warp, lane);
            }
            // dX of this tile, added to the row's gradient
            wait_or_fail(dxready, g & 1, failed, status);
            tc_fence_after();
            constexpr int HC = C::d / 4;  // columns per thread
            uint32_t x[HC];
            if constexpr (HC == 8) tmem_ld8(tbase + lrow + cX + H * HC, x);
            else tmem_ld16(tbase + lrow + cX + H * HC, x);
            tmem_wait_ld();
            tc_fence_before();
            mbar_arrive(dxfree);
            if (valid) {
                uint4 *row = reinterpret_cast<uint4 *>(dXg + ((size_t)bh * a.n + row0 + r) * C::d + H * HC);
#pragma unroll
                for (int k = 0; k < HC / 8; ++k) {
                    const uint4 old = row[k];
                    const uint32_t ow[4] = {old.x, old.y, old.z, old.w};
                    float f[8];
#pragma unroll
                    for (int c = 0; c < 4; ++c) {
                        f[2 * c] = __uint_as_float(ow[c] << 16) + __uint_as_float(x[8 * k + 2 * c]);
                        f[2 * c + 1] = __uint_as_float(ow[c] & 0xffff0000u) + __uint_as_float(x[8 * k + 2 * c + 1]);
                    }
                    row[k] = pack8(f);
                }
            }
            ++g;
        }
        if (hacc.tiles > 0) hist_close(bins, hpart, a.lay.nint, hacc, tid, false, smax, warp, lane);
#pragma unroll
        for (int q = 0; q < PP; ++q) {
            float v = db_acc[q];
#pragma unroll
            for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
            if (lane == 0) atomicAdd(sdb + H * PP + q, v);
        }
        // dW^T accumulator (M = 64: input column cd in lane 32*(cd/16) + cd%16)
        if (warp < 4) {
            const bool any = g > 0;
            if (any) wait_or_fail(wdone, 0, failed, status);
            tc_fence_after();
            uint32_t xw[16];
            tmem_ld16(tbase + ((uint32_t)(warp << 5) << 16) + cW, xw);
            tmem_wait_ld();
            const int cd = (warp << 4) | lane;
            if (any && lane < 16 && cd < C::d)
#pragma unroll
                for (int i = 0; i < C::MP; ++i) sdW[i * C::d + cd] = __uint_as_float(xw[i]) + __uint_as_float(xw[C::MP + i]);
        }
    }
    tc_fence_before();
    __syncthreads();
    store_param_partial<C>(a, sdW, sdb, gp);
    __syncthreads();
    if (warp == 0) tmem_dealloc(tbase, 256);
}

template <class C>
cudaError_t kterm_tc_impl(const AttnArgs &a, float *gpart, int grid, cudaStream_t s) {
    CUtensorMap mQ, mK;
    if (!tc_make_map(&mQ, a.Q, a.d, a.n, a.B * a.H, 1) || !tc_make_map(&mK, a.K, a.d, a.n, a.B * a.H, 1))
        return cudaErrorInvalidValue;
    cudaError_t e = cudaFuncSetAttribute(k_tc_kterm<C>, cudaFuncAttributeMaxDynamicSharedMemorySize, C::SMEM);
    if (e != cudaSuccess) return e;
    int *st = reinterpret_cast<int *>(reinterpret_cast<char *>(a.counters) - 256);  // the workspace status word
    LUNA_LAUNCH("tc_kterm", k_tc_kterm<C>, dim3(grid, 2), kBThreads, C::SMEM, s, mQ, mK, a, a.ch_kappa, gpart, st);
    return cudaGetLastError();
}

}  // namespace

// The scale-term pass on tensor cores for bf16, d = 32 or 64, M = 8, L = 8, fp32 partials (the
// non-causal tensor-core backward), 16-byte aligned tensors; false: the caller runs the CUDA-core pass.
bool tc_kterm_supported(const AttnArgs &a) {
    auto al = [](const void *x) { return (reinterpret_cast<uintptr_t>(x) & 15) == 0; };
    return !a.gpart64 && a.ch_io == LUNA_BF16 && a.L == 8 && a.M == 8 && (a.d == 32 || a.d == 64) &&
           a.lay.P <= kPpad && a.hs_mul == 1 && !a.lay.signed_out && al(a.Q) && al(a.K) && al(a.dQ) && al(a.dK);
}

// Launches it with at most max_parts blocks per side; *nparts: the partials per side.
cudaError_t launch_tc_kterm(const AttnArgs &a, float *gpart, int max_parts, int *nparts, cudaStream_t s) {
    int grid = tc_sm_count() / 2;
    grid = grid < 1 ? 1 : (grid > max_parts ? max_parts : grid);
    *nparts = grid;
    return a.d == 32 ? kterm_tc_impl<KCfg<32>>(a, gpart, grid, s) : kterm_tc_impl<KCfg<64>>(a, gpart, grid, s);
}

}  // namespace luna
