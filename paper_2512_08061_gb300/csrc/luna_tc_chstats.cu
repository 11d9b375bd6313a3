// Channel RMS statistics on tensor cores (bf16 I/O, the tensor-core shapes):
// the sums over every valid row and projection of phi_l^2, for the queries
// (blockIdx.y = 0) and the keys (blockIdx.y = 1), as block partials
// part[(side * gridDim.x + blockIdx.x) * L + l] in the layout of the CUDA-core
// statistics pass, which the scale kernel then reduces.
//
// Per 128-row tile (warp roles as in the forward kernels):
//   TMA   X tile into one of four stages
//   MMA   U = X [W_hi; W_mid]^T into one of two TMEM buffers
//   work  u, interval (bucketed search block), phi of the 8 channels from the interval table, sum of
//         phi^2 per channel in registers (rows past a sequence's length add nothing)
// The tiles of a side are dealt to the blocks round robin; every role walks the same sequence.
#include "luna_tc_dev.cuh"

namespace luna {

bool tc_make_map(CUtensorMap *m, const void *base, int width, int n, int BH, int hs_mul);
int tc_sm_count();

namespace {
using namespace sm100;
using namespace simt;
using namespace tcdev;

constexpr int kSWorkers = 512;  // 16 warps, four threads per row
constexpr int kSTma = 16, kSMma = 17;
constexpr int kSThreads = kSWorkers + 64;

template <int DX_, int MP_>
struct SCfg {
    static constexpr int DX = DX_, MP = MP_, NU = 2 * MP, KBX = DX / 64, PP = MP / 4;
    static constexpr uint32_t XT = 128u * DX * 2;        // X tile
    static constexpr uint32_t WOP = (uint32_t)NU * DX * 2;  // [W_hi; W_mid] operand
    static constexpr int NX = 4;
    static constexpr uint32_t RED = (kSWorkers / 32) * 8 * 4;
    static constexpr uint32_t SMEM = NX * XT + WOP + kTableBytes + 32 * 4 + RED + 256 + 1024;
    static constexpr uint32_t TMEM = 2 * NU <= 32 ? 32 : 2 * NU <= 64 ? 64 : 128;
    static_assert(SMEM <= kSmemLimit, "shared memory budget");
    static_assert(PP == 2 || PP == 4, "projections per worker");
};

// Tile t of a side: row0 = (t % nt) * 128 of head t / nt; it holds valid rows iff row0 < the head's length.
__device__ __forceinline__ bool tile_live(const AttnArgs &a, int64_t t, int nt, int &row0, int &bh) {
    bh = (int)(t / nt);
    row0 = (int)(t - (int64_t)bh * nt) * 128;
    return row0 < head_length(a.lengths, bh / a.H, a.n);
}

template <class C>
__global__ void __launch_bounds__(kSThreads, 1)
    k_tc_chstats(const __grid_constant__ CUtensorMap mapQ, const __grid_constant__ CUtensorMap mapK, AttnArgs a,
                 float *part, int *status) {
    extern __shared__ uint8_t smem_raw[];
    uint8_t *sm = align1024(smem_raw);
    constexpr int NX = C::NX, PP = C::PP;
    uint8_t *Xb = sm;
    uint8_t *Wop = Xb + NX * C::XT;
    float *sTe = reinterpret_cast<float *>(Wop + C::WOP);
    float *sAB = sTe + kEytzinger;
    float *sbias = sAB + kNint * 16;
    float *sred = sbias + 32;  // [worker warps][8]
    uint64_t *bars = reinterpret_cast<uint64_t *>(sred + C::RED / 4);
    uint64_t *fullx = bars;         // [NX] X tile landed
    uint64_t *xfree = fullx + NX;   // [NX] projection consumed it
    uint64_t *uready = xfree + NX;  // [2] projection in TMEM
    uint64_t *ufree = uready + 2;   // [2] workers read it (count 512)
    uint32_t *tslot = reinterpret_cast<uint32_t *>(ufree + 2);
    static_assert((2 * NX + 4) * 8 + 4 <= 256, "barrier area");

    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int side = blockIdx.y;
    const int nt = (a.n + 127) / 128;
    const int64_t tiles = (int64_t)a.B * a.H * nt;
    if (tid == 0) {
        for (int i = 0; i < NX; ++i) { mbar_init(fullx + i, 1); mbar_init(xfree + i, 1); }
        for (int i = 0; i < 2; ++i) { mbar_init(uready + i, 1); mbar_init(ufree + i, kSWorkers); }
        fence_mbar_init();
    }
    if (warp == 0) { tmem_alloc(tslot, C::TMEM); tmem_relinquish(); }
    stage_phi_table<C>(a, sTe, sAB, sbias, Wop);
    fence_proxy_async_smem();
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tbase = *tslot;

    if (warp == kSTma) {
        if (lane == 0) {
            const CUtensorMap *map = side ? &mapK : &mapQ;
            bool failed = false;
            int g = 0, row0, bh;
            for (int64_t t = blockIdx.x; t < tiles && !failed; t += gridDim.x) {
                if (!tile_live(a, t, nt, row0, bh)) continue;
                const int x = g % NX;
                if (g >= NX) wait_or_fail(xfree + x, ((g - NX) / NX) & 1, failed, status);
                mbar_arrive_expect_tx(fullx + x, C::XT);
                for (int kb = 0; kb < C::KBX; ++kb) tma_load_3d(Xb + x * C::XT + kb * 16384, map, kb * 64, row0, bh, fullx + x);
                ++g;
            }
        }
    } else if (warp == kSMma) {
        if (lane == 0) {
            const uint64_t dx0 = sdesc(smem_u32(Xb), 16, 1024, kSwizzle128);
            const uint64_t dw0 = sdesc(smem_u32(Wop), 16, 1024, kSwizzle128);
            constexpr uint32_t idU = idesc_bf16(128, C::NU, false, false);
            bool failed = false;
            int g = 0, row0, bh;
            for (int64_t t = blockIdx.x; t < tiles && !failed; t += gridDim.x) {
                if (!tile_live(a, t, nt, row0, bh)) continue;
                const int x = g % NX, b = g & 1;
                wait_or_fail(fullx + x, (g / NX) & 1, failed, status);
                if (g >= 2) wait_or_fail(ufree + b, ((g - 2) >> 1) & 1, failed, status);
                tc_fence_after();
#pragma unroll
                for (int kb = 0; kb < C::KBX; ++kb)
#pragma unroll
                    for (int k = 0; k < 4; ++k)
                        mma_bf16_ss(tbase + b * C::NU, dadd(dx0, x * C::XT + kb * 16384 + 32 * k),
                                    dadd(dw0, kb * (C::NU * 128) + 32 * k), idU, (kb | k) != 0);
                mma_commit(uready + b);
                mma_commit(xfree + x);
                ++g;
            }
        }
    } else {
        // workers: thread (Q, r) owns row r of the tile and projections Q*PP .. Q*PP+PP-1
        const int Q = warp >> 2, r = ((warp & 3) << 5) | lane;
        const uint32_t lrow = (uint32_t)((warp & 3) << 5) << 16;
        bool failed = false;
        float acc[8] = {};
        int g = 0, row0, bh;
        for (int64_t t = blockIdx.x; t < tiles; t += gridDim.x) {
            if (!tile_live(a, t, nt, row0, bh)) continue;
            const int b = g & 1;
            const bool valid = row0 + r < head_length(a.lengths, bh / a.H, a.n);
            wait_or_fail(uready + b, (g >> 1) & 1, failed, status);
            tc_fence_after();
            float u[PP];
            {
                uint32_t xh[PP], xl[PP];
                const uint32_t col = tbase + lrow + b * C::NU + Q * PP;
                if constexpr (PP == 2) {
                    tmem_ld2(col, xh);
                    tmem_ld2(col + C::MP, xl);
                } else {
                    tmem_ld4(col, xh);
                    tmem_ld4(col + C::MP, xl);
                }
                tmem_wait_ld();
#pragma unroll
                for (int q = 0; q < PP; ++q)
                    u[q] = __uint_as_float(xh[q]) + __uint_as_float(xl[q]) + sbias[Q * PP + q];
            }
            tc_fence_before();
            mbar_arrive(ufree + b);  // the buffer may take the projection two tiles on
            ++g;
            if (!valid) continue;
            int j[PP];
            search_bucketed<PP>(sTe, u, j);
            const float4 *ab = reinterpret_cast<const float4 *>(sAB);
#pragma unroll
            for (int q = 0; q < PP; ++q)
#pragma unroll
                for (int k = 0; k < 4; ++k) {
                    const float4 v = ab[ab_slot(j[q], k)];
                    const float y0 = fmaxf(fmaf(v.x, u[q], v.y), 0.0f), y1 = fmaxf(fmaf(v.z, u[q], v.w), 0.0f);
                    acc[2 * k] = fmaf(y0, y0, acc[2 * k]);
                    acc[2 * k + 1] = fmaf(y1, y1, acc[2 * k + 1]);
                }
        }
        // block sums: lanes, then the worker warps in order
#pragma unroll
        for (int l = 0; l < 8; ++l) {
            float v = acc[l];
#pragma unroll
            for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
            if (lane == 0) sred[warp * 8 + l] = v;
        }
        named_sync<kSWorkers>(1);
        if (tid < 8) {
            float v = 0.0f;
            for (int w = 0; w < kSWorkers / 32; ++w) v += sred[w * 8 + tid];
            part[((size_t)side * gridDim.x + blockIdx.x) * 8 + tid] = v;
        }
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 0) tmem_dealloc(tbase, C::TMEM);
}

template <class C>
cudaError_t chstats_impl(const AttnArgs &a, float *part, int grid, cudaStream_t s) {
    CUtensorMap mQ, mK;
    if (!tc_make_map(&mQ, a.Q, a.d, a.n, a.B * a.H, 1) || !tc_make_map(&mK, a.K, a.d, a.n, a.B * a.H, 1))
        return cudaErrorInvalidValue;
    cudaError_t e = cudaFuncSetAttribute(k_tc_chstats<C>, cudaFuncAttributeMaxDynamicSharedMemorySize, C::SMEM);
    if (e != cudaSuccess) return e;
    int *st = reinterpret_cast<int *>(reinterpret_cast<char *>(a.counters) - 256);  // the workspace status word
    LUNA_LAUNCH("tc_chstats", k_tc_chstats<C>, dim3(grid, 2), kSThreads, C::SMEM, s, mQ, mK, a, part, st);
    return cudaGetLastError();
}

}  // namespace

// The statistics of both sides on tensor cores for the shapes of the forward tensor-core kernels (bf16,
// L = 8, (d, M) = (32, 8), (64, 8), (128, 16), 16-byte aligned inputs); false when the shape is not one
// of them (the caller runs the CUDA-core pass).  *nparts: the partials per side.
bool tc_chstats_supported(const AttnArgs &a, luna_dtype io) {
    auto al = [](const void *x) { return (reinterpret_cast<uintptr_t>(x) & 15) == 0; };
    if (io != LUNA_BF16 || a.L != 8 || a.lay.P > kPpad || a.hs_mul != 1 || a.lay.signed_out || !al(a.Q) || !al(a.K))
        return false;
    return (a.M == 8 && (a.d == 32 || a.d == 64)) || (a.M == 16 && a.d == 128);
}

cudaError_t launch_tc_chstats(const AttnArgs &a, float *part, int max_parts, int *nparts, cudaStream_t s) {
    int grid = tc_sm_count() / 2;  // two sides: one block per SM
    grid = grid < 1 ? 1 : (grid > max_parts ? max_parts : grid);
    *nparts = grid;
    return a.M == 16 ? chstats_impl<SCfg<128, 16>>(a, part, grid, s) : chstats_impl<SCfg<64, 8>>(a, part, grid, s);
}

}  // namespace luna
