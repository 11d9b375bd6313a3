// Tensor-core (tcgen05 / TMEM / TMA) kernels for bf16 I/O on sm_103a.
//
// Every kernel works on tiles of 128 rows of one (batch, head) with 288
// threads: warp 8 is the producer (one elected lane issues the TMA tile loads
// and the tcgen05.mma instructions and commits them to mbarriers); warps 0..7
// are workers, two per row (warps w and w+4 own TMEM lanes 32*(w%4)..+31 and
// split the M projections of those rows between them).
//
// Per tile, forward key pass (Sec. 4, S_KV and S_K1):
//   TMA K, V -> smem (128B swizzle)
//   MMA  U = K [W_hi; W_lo]^T                      (projections, TMEM)
//   workers: u = U_hi + U_lo + b; interval j of u in the merged kink list;
//            phi = relu(alpha_j u + beta_j) for the 8 channels -> bf16 tile
//   MMA  S += phi^T V,  z += phi^T 1               (MN-major A and B, TMEM)
// Forward query pass (Eq. kernel-attn):
//   TMA Q -> MMA U -> phi tile + fp32 normaliser phi.z
//   MMA  num = phi [S_hi; S_lo]^T,  O = num / (phi.z + eps)
// S is split into bf16 hi + lo parts so that the state enters the product with
// ~16 significant bits; W likewise.  phi itself is rounded to bf16.
#include <math.h>
#include <stdlib.h>

#include "luna_prof.cuh"
#include "luna_sm100.cuh"
#include "luna_simt_dev.cuh"
#include "luna_tc.cuh"

namespace luna {
namespace {
using namespace sm100;
using namespace simt;

constexpr int kWorkers = 256;
constexpr int kThreadsTC = kWorkers + 32;
constexpr uint32_t kSmemLimit = 227 * 1024;
constexpr int kPpad = 512;   // merged kink list (L * hidden <= 512, L = 8)
constexpr int kNint = 513;   // intervals

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
    static constexpr int PP = MP / 2;             // projections per worker thread
    static constexpr int NUS = 2;                 // projection stages in TMEM
    static constexpr uint32_t XT = 128u * DX * 2;
    static constexpr uint32_t VT = 128u * VC * 2;
    static constexpr uint32_t PT = 128u * D * 2;  // one bf16 phi tile
    static constexpr uint32_t WOP = (uint32_t)NU * DX * 2;
    static constexpr uint32_t ONES = 4096;
    static constexpr uint32_t TABLE = (kPpad + kNint * 16 + 32) * 4;
    static constexpr uint32_t MISC = 1024;
    static constexpr bool SMALL = XT <= 16384 && VT <= 16384;
    // key pass: phi(K) as bf16 hi + lo tiles
    static constexpr int NX_K = SMALL ? 3 : 2;
    static constexpr int NV_K = SMALL ? 3 : 1;
    static constexpr int NP_K = SMALL ? 2 : 1;
    static constexpr uint32_t FIX_K = WOP + ONES + TABLE + MISC + 1024;
    static constexpr uint32_t SMEM_K = NX_K * XT + NV_K * VT + NP_K * 2 * PT + FIX_K;
    static constexpr int TMEM_K_USED = NU * NUS + DV + 16;
    static constexpr int TMEM_K = TMEM_K_USED <= 32 ? 32 : TMEM_K_USED <= 64 ? 64 : TMEM_K_USED <= 128 ? 128
                                 : TMEM_K_USED <= 256 ? 256 : 512;
    // query pass: phi(Q) as one bf16 tile
    static constexpr uint32_t SOP = 2u * DV * D * 2;  // [S_hi; S_lo]^T operand
    static constexpr int NP_Q = SMALL ? 2 : 1;
    static constexpr int NX_Q = SMALL ? 4 : 2;
    static constexpr uint32_t FIX_Q = WOP + SOP + TABLE + D * 4 + 2 * 2 * 128 * 4 + MISC + 1024;
    static constexpr uint32_t SMEM_Q = NX_Q * XT + NP_Q * PT + FIX_Q;
    static constexpr int NN_Q = (NU * NUS + 4 * DV <= 256) ? 2 : 1;
    static constexpr int TMEM_Q_USED = NU * NUS + 2 * DV * NN_Q;
    static constexpr int TMEM_Q = TMEM_Q_USED <= 64 ? 64 : TMEM_Q_USED <= 128 ? 128 : TMEM_Q_USED <= 256 ? 256 : 512;
    static_assert(SMEM_K <= kSmemLimit && SMEM_Q <= kSmemLimit, "shared memory budget");
    static_assert(TMEM_K_USED <= 512 && TMEM_Q_USED <= 512, "tensor memory budget");
};

__device__ __forceinline__ uint8_t *align1024(uint8_t *p) {
    return reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(p) + 1023) & ~uintptr_t(1023));
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

// Loads the kink list, the interval table and the projection bias into smem,
// and writes the projection operand [W_hi; W_lo] (NU rows x DX, K-major SW128).
template <class C>
__device__ void stage_phi_table(const AttnArgs &a, float *sT, float *sAB, float *sbias, uint8_t *Wop, int tid,
                                int nthreads) {
    const TableLayout &lay = a.lay;
    const float *T = reinterpret_cast<const float *>(a.table + lay.off_T);
    for (int e = tid; e < kPpad; e += nthreads) sT[e] = e < lay.Ppad ? T[e] : INFINITY;
    const float4 *AB4 = reinterpret_cast<const float4 *>(a.table + lay.off_AB);
    for (int e = tid; e < lay.nint * 4; e += nthreads) reinterpret_cast<float4 *>(sAB)[e] = AB4[e];
    const float *b = reinterpret_cast<const float *>(a.table + lay.off_b);
    for (int e = tid; e < C::MP; e += nthreads) sbias[e] = b[e];
    const float *W = reinterpret_cast<const float *>(a.table + lay.off_W);
    for (int e = tid; e < C::NU * C::DX; e += nthreads) {
        const int n = e / C::DX, c = e % C::DX;
        const int i = n % C::MP;
        const float w = (c < a.d) ? W[i * a.d + c] : 0.0f;
        __nv_bfloat16 hi, lo;
        split_bf16(w, hi, lo);
        *reinterpret_cast<__nv_bfloat16 *>(Wop + (c / 64) * (C::NU * 128) + sw128_chunk(n, (c % 64) / 8) + (c % 8) * 2) =
            (n < C::MP) ? hi : lo;
    }
}

// Projection MMA: U[cols] = X tile (128 x DX) * [W_hi; W_lo]^T
template <class C>
__device__ __forceinline__ void issue_proj(uint32_t tmem_u, uint32_t xaddr, uint32_t waddr) {
    constexpr uint32_t idesc = idesc_bf16(128, C::NU, false, false);
#pragma unroll
    for (int kb = 0; kb < C::KBX; ++kb)
#pragma unroll
        for (int k = 0; k < 4; ++k)
            mma_bf16_ss(tmem_u, sdesc(xaddr + kb * 16384 + 32 * k, 16, 1024, kSwizzle128),
                        sdesc(waddr + kb * (C::NU * 128) + 32 * k, 16, 1024, kSwizzle128), idesc, (kb | k) != 0);
}

// Worker: phi for projections [H*PP, H*PP+PP) of row r from the projection
// columns in TMEM; writes the bf16 chunks of the phi tile (and, if plo is not
// null, the bf16 residual phi - bf16(phi) into a second tile), zeros for rows
// that are not valid; optionally accumulates the fp32 normaliser phi . z.
template <class C, int H>
__device__ __forceinline__ void phi_row_half(uint32_t tmem_u_row, const float *sT, const float *sAB,
                                             const float *sbias, bool valid, int r, uint8_t *phi, uint8_t *plo,
                                             const float *sz, float &den) {
    uint32_t hv[C::PP], lv[C::PP];
    if constexpr (C::PP == 4) {
        uint32_t x[16];
        tmem_ld16(tmem_u_row, x);
        tmem_wait_ld();
#pragma unroll
        for (int q = 0; q < 4; ++q) { hv[q] = x[H * 4 + q]; lv[q] = x[8 + H * 4 + q]; }
    } else {
        uint32_t x[16], y[16];
        tmem_ld16(tmem_u_row, x);
        tmem_ld16(tmem_u_row + 16, y);
        tmem_wait_ld();
#pragma unroll
        for (int q = 0; q < 8; ++q) { hv[q] = x[H * 8 + q]; lv[q] = y[H * 8 + q]; }
    }
#pragma unroll
    for (int q = 0; q < C::PP; ++q) {
        constexpr int base = H * C::PP;
        const int i = base + q;
        uint4 ph = make_uint4(0u, 0u, 0u, 0u), pl = make_uint4(0u, 0u, 0u, 0u);
        if (valid) {
            const float u = __uint_as_float(hv[q]) + __uint_as_float(lv[q]) + sbias[i];
            const int j = interval_of(sT, kPpad, u);
            const float4 *ab = reinterpret_cast<const float4 *>(sAB) + j * 4;
            float y[8];
#pragma unroll
            for (int k = 0; k < 4; ++k) {
                const float4 v = ab[k];
                y[2 * k] = fmaxf(fmaf(v.x, u, v.y), 0.0f);
                y[2 * k + 1] = fmaxf(fmaf(v.z, u, v.w), 0.0f);
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

template <int N>
__device__ __forceinline__ void named_sync(int id) {
    asm volatile("bar.sync %0, %1;" ::"r"(id), "r"(N) : "memory");
}

// ---------------------------------------------------------------------------
// forward key pass: S_KV = phi(K)^T V and S_K1 = phi(K)^T 1 per (head, split)
//
// phi(K) enters the contraction as bf16 hi + lo tiles (two MMAs), so that the
// key statistics carry ~16 significant bits of phi: the backward pass
// subtracts nearly equal terms built from S and z.

template <class C>
__global__ void __launch_bounds__(kThreadsTC, 1)
    k_tc_keys(const __grid_constant__ CUtensorMap mapK, const __grid_constant__ CUtensorMap mapV, AttnArgs a,
              int *status) {
    extern __shared__ uint8_t smem_raw[];
    uint8_t *sm = align1024(smem_raw);
    constexpr int NX = C::NX_K, NV = C::NV_K, NP = C::NP_K, NUS = C::NUS;
    uint8_t *Xb = sm;
    uint8_t *Vb = Xb + NX * C::XT;
    uint8_t *Pb = Vb + NV * C::VT;  // [NP][hi, lo]
    uint8_t *Wop = Pb + NP * 2 * C::PT;
    uint8_t *Ones = Wop + C::WOP;
    float *sT = reinterpret_cast<float *>(Ones + C::ONES);
    float *sAB = sT + kPpad;
    float *sbias = sAB + kNint * 16;
    uint64_t *bars = reinterpret_cast<uint64_t *>(sbias + 32);
    uint64_t *fullx = bars;            // [NX] X tile landed
    uint64_t *xfree = fullx + NX;      // [NX] projection MMA consumed it
    uint64_t *fullv = xfree + NX;      // [NV] V tile landed
    uint64_t *vfree = fullv + NV;      // [NV] contraction consumed it
    uint64_t *uready = vfree + NV;     // [NUS] projection in TMEM
    uint64_t *phiready = uready + NUS; // [NP] workers wrote phi (count 256)
    uint64_t *pfree = phiready + NP;   // [NP] contraction consumed phi
    uint64_t *accdone = pfree + NP;    // [1]
    uint32_t *tslot = reinterpret_cast<uint32_t *>(accdone + 1);

    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int bh = blockIdx.y, split = blockIdx.x;
    const int len = head_length(a.lengths, bh / a.H, a.n);
    const int r0 = split * a.rows_per_split;
    const int r1 = min(len, r0 + a.rows_per_split);
    const int ntiles = r1 > r0 ? (r1 - r0 + 127) / 128 : 0;

    if (tid == 0) {
        for (int i = 0; i < NX; ++i) { mbar_init(fullx + i, 1); mbar_init(xfree + i, 1); }
        for (int i = 0; i < NV; ++i) { mbar_init(fullv + i, 1); mbar_init(vfree + i, 1); }
        for (int i = 0; i < NUS; ++i) mbar_init(uready + i, 1);
        for (int i = 0; i < NP; ++i) { mbar_init(phiready + i, kWorkers); mbar_init(pfree + i, 1); }
        mbar_init(accdone, 1);
        fence_mbar_init();
    }
    if (warp == 0) { tmem_alloc(tslot, C::TMEM_K); tmem_relinquish(); }
    stage_phi_table<C>(a, sT, sAB, sbias, Wop, tid, kThreadsTC);
    for (int e = tid; e < (int)C::ONES / 4; e += kThreadsTC)
        reinterpret_cast<uint32_t *>(Ones)[e] = 0x3F803F80u;  // bf16 1.0 pairs
    fence_proxy_async_smem();
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tbase = *tslot;
    const uint32_t tmem_s = tbase + C::NU * NUS;  // S accumulator (DV cols)
    const uint32_t tmem_z = tmem_s + C::DV;       // z accumulator (16 cols)

    if (warp == 8) {
        if (lane == 0 && ntiles > 0) {
            const uint32_t xa = smem_u32(Xb), va = smem_u32(Vb), pa = smem_u32(Pb), wa = smem_u32(Wop),
                           oa = smem_u32(Ones);
            auto load_x = [&](int t) {
                const int x = t % NX;
                mbar_arrive_expect_tx(fullx + x, C::XT);
                for (int kb = 0; kb < C::KBX; ++kb)
                    tma_load_3d(Xb + x * C::XT + kb * 16384, &mapK, kb * 64, r0 + t * 128, bh, fullx + x);
            };
            auto load_v = [&](int t) {
                const int v = t % NV;
                mbar_arrive_expect_tx(fullv + v, C::VT);
                for (int vb = 0; vb < C::NVB; ++vb)
                    tma_load_3d(Vb + v * C::VT + vb * 16384, &mapV, vb * 64, r0 + t * 128, bh, fullv + v);
            };
            auto proj = [&](int t) {
                const int x = t % NX;
                issue_proj<C>(tbase + (t % NUS) * C::NU, xa + x * C::XT, wa);
                mma_commit(uready + (t % NUS));
                mma_commit(xfree + x);
            };
            bool failed = false;
            for (int t = 0; t < NX && t < ntiles; ++t) load_x(t);
            for (int t = 0; t < NV && t < ntiles; ++t) load_v(t);
            wait_or_fail(fullx, 0, failed, status);
            tc_fence_after();
            proj(0);
            for (int t = 0; t < ntiles && !failed; ++t) {
                const int p = t % NP, v = t % NV;
                if (t + 1 < ntiles) {
                    wait_or_fail(fullx + (t + 1) % NX, ((t + 1) / NX) & 1, failed, status);
                    tc_fence_after();
                    proj(t + 1);
                }
                if (t + NX < ntiles) {
                    wait_or_fail(xfree + t % NX, (t / NX) & 1, failed, status);
                    load_x(t + NX);
                }
                wait_or_fail(phiready + p, (t / NP) & 1, failed, status);
                wait_or_fail(fullv + v, (t / NV) & 1, failed, status);
                tc_fence_after();
                const uint32_t ph = pa + p * 2 * C::PT, pl = ph + C::PT, vt = va + v * C::VT;
                constexpr uint32_t idS = idesc_bf16(C::D, C::DV, true, true);
                constexpr uint32_t idZ = idesc_bf16(C::D, 16, true, false);
#pragma unroll
                for (int k = 0; k < 8; ++k) {
                    const uint32_t acc = (t > 0 || k > 0) ? 1u : 0u;
                    const uint64_t bv = sdesc(vt + 2048 * k, 16384, 1024, kSwizzle128);
                    const uint64_t bo = sdesc(oa + (k / 4) * 2048 + 32 * (k % 4), 16, 1024, kSwizzle128);
                    const uint64_t ah = sdesc(ph + 2048 * k, 16384, 1024, kSwizzle128);
                    const uint64_t al = sdesc(pl + 2048 * k, 16384, 1024, kSwizzle128);
                    mma_bf16_ss(tmem_s, ah, bv, idS, acc);
                    mma_bf16_ss(tmem_s, al, bv, idS, 1u);
                    mma_bf16_ss(tmem_z, ah, bo, idZ, acc);
                    mma_bf16_ss(tmem_z, al, bo, idZ, 1u);
                }
                mma_commit(pfree + p);
                mma_commit(vfree + v);
                if (t + NV < ntiles) {
                    wait_or_fail(vfree + v, (t / NV) & 1, failed, status);
                    load_v(t + NV);
                }
            }
            if (!failed) mma_commit(accdone);
            else mbar_arrive(accdone);
        }
    } else {
        const int h = warp >> 2, r = ((warp & 3) << 5) | lane;
        const uint32_t lrow = (uint32_t)((warp & 3) << 5) << 16;
        float dummy = 0.0f;
        bool failed = false;
        for (int t = 0; t < ntiles; ++t) {
            const int p = t % NP, v = t % NV;
            const int nvalid = min(128, r1 - (r0 + t * 128));
            wait_or_fail(uready + t % NUS, (t / NUS) & 1, failed, status);
            if (t >= NP) wait_or_fail(pfree + p, ((t - NP) / NP) & 1, failed, status);
            tc_fence_after();
            uint8_t *ph = Pb + p * 2 * C::PT, *pl = ph + C::PT;
            const bool valid = r < nvalid;
            const uint32_t ucol = tbase + lrow + (t % NUS) * C::NU;
            if (h == 0) phi_row_half<C, 0>(ucol, sT, sAB, sbias, valid, r, ph, pl, nullptr, dummy);
            else phi_row_half<C, 1>(ucol, sT, sAB, sbias, valid, r, ph, pl, nullptr, dummy);
            if (!valid && h == 0) {  // padded rows: clear V so that no garbage enters S
                wait_or_fail(fullv + v, (t / NV) & 1, failed, status);
                uint8_t *vrow = Vb + v * C::VT;
#pragma unroll
                for (int vb = 0; vb < C::NVB; ++vb)
#pragma unroll
                    for (int c = 0; c < 8; ++c)
                        *reinterpret_cast<uint4 *>(vrow + vb * 16384 + sw128_chunk(r, c)) = make_uint4(0, 0, 0, 0);
            }
            fence_proxy_async_smem();
            tc_fence_before();
            mbar_arrive(phiready + p);
        }
    }
    // epilogue: partial S, z of this split -> workspace; the last split reduces
    const size_t slot = (size_t)bh * a.nsplit + split;
    float *Sp = a.S_part + slot * C::D * C::DV;
    float *zp = a.z_part + slot * C::D;
    if (warp < 4) {
        bool failed = false;
        if (ntiles > 0) wait_or_fail(accdone, 0, failed, status);
        const bool ok = !failed && ntiles > 0;
        tc_fence_after();
        // accumulator row f: M = 128 -> TMEM lane f; M = 64 -> lane 32*(f/16) + f%16
        const int f = (C::D == 128) ? ((warp << 5) | lane) : ((warp << 4) | lane);
        const bool holds = (C::D == 128) || lane < 16;
        const uint32_t lrow = (uint32_t)(warp << 5) << 16;
#pragma unroll
        for (int c0 = 0; c0 < C::DV; c0 += 16) {
            uint32_t x[16];
            tmem_ld16(lrow + tmem_s + c0, x);
            tmem_wait_ld();
            if (holds) {
#pragma unroll
                for (int c = 0; c < 16; c += 4)
                    *reinterpret_cast<float4 *>(Sp + f * C::DV + c0 + c) =
                        ok ? make_float4(__uint_as_float(x[c]), __uint_as_float(x[c + 1]), __uint_as_float(x[c + 2]),
                                         __uint_as_float(x[c + 3]))
                           : make_float4(0.f, 0.f, 0.f, 0.f);
            }
        }
        uint32_t x[16];
        tmem_ld16(lrow + tmem_z, x);
        tmem_wait_ld();
        if (holds) zp[f] = ok ? __uint_as_float(x[0]) : 0.0f;
    }
    tc_fence_before();
    if (last_arrival(a.counters + bh, a.nsplit)) {
        ordered_sum(a.S_part + (size_t)bh * a.nsplit * C::D * C::DV, a.nsplit, C::D * C::DV,
                    a.S_fin + (size_t)bh * C::D * C::DV);
        ordered_sum(a.z_part + (size_t)bh * a.nsplit * C::D, a.nsplit, C::D, a.z_fin + (size_t)bh * C::D);
        if (tid == 0) a.counters[bh] = 0;
    }
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
    constexpr int NX = C::NX_Q, NP = C::NP_Q, NN = C::NN_Q, NUS = C::NUS;
    uint8_t *Xb = sm;
    uint8_t *Pb = Xb + NX * C::XT;
    uint8_t *Wop = Pb + NP * C::PT;
    uint8_t *Sop = Wop + C::WOP;
    float *sT = reinterpret_cast<float *>(Sop + C::SOP);
    float *sAB = sT + kPpad;
    float *sbias = sAB + kNint * 16;
    float *sz = sbias + 32;
    float *sden = sz + C::D;  // [2 tiles][2 halves][128 rows]
    uint64_t *bars = reinterpret_cast<uint64_t *>(sden + 512);
    uint64_t *fullx = bars;               // [NX]
    uint64_t *xfree = fullx + NX;         // [NX]
    uint64_t *uready = xfree + NX;        // [NUS]
    uint64_t *phiready = uready + NUS;    // [NP] count 256
    uint64_t *pfree = phiready + NP;      // [NP]
    uint64_t *numready = pfree + NP;      // [NN]
    uint64_t *numfree = numready + NN;    // [NN] count 256
    uint32_t *tslot = reinterpret_cast<uint32_t *>(numfree + NN);

    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int bh = blockIdx.y, split = blockIdx.x;
    const int len = head_length(a.lengths, bh / a.H, a.n);
    const int r0 = split * a.rows_per_split;
    const int rend = min(a.n, r0 + a.rows_per_split);
    const int r1 = min(len, rend);
    const int ntiles = r1 > r0 ? (r1 - r0 + 127) / 128 : 0;
    __nv_bfloat16 *O = static_cast<__nv_bfloat16 *>(a.O) + (size_t)bh * a.n * C::DV;

    if (tid == 0) {
        for (int i = 0; i < NX; ++i) { mbar_init(fullx + i, 1); mbar_init(xfree + i, 1); }
        for (int i = 0; i < NUS; ++i) mbar_init(uready + i, 1);
        for (int i = 0; i < NP; ++i) { mbar_init(phiready + i, kWorkers); mbar_init(pfree + i, 1); }
        for (int i = 0; i < NN; ++i) { mbar_init(numready + i, 1); mbar_init(numfree + i, kWorkers); }
        fence_mbar_init();
    }
    if (warp == 0) { tmem_alloc(tslot, C::TMEM_Q); tmem_relinquish(); }
    stage_phi_table<C>(a, sT, sAB, sbias, Wop, tid, kThreadsTC);
    const float *Sg = a.S_fin + (size_t)bh * C::D * C::DV;
    for (int e = tid; e < 2 * C::DV * C::D; e += kThreadsTC) {
        const int n = e / C::D, f = e % C::D;  // operand row n: output column n % DV, hi (n < DV) or lo part
        __nv_bfloat16 hi, lo;
        split_bf16(Sg[f * C::DV + (n % C::DV)], hi, lo);
        *reinterpret_cast<__nv_bfloat16 *>(Sop + (f / 64) * (2 * C::DV * 128) + sw128_chunk(n, (f % 64) / 8) +
                                           (f % 8) * 2) = (n < C::DV) ? hi : lo;
    }
    for (int e = tid; e < C::D; e += kThreadsTC) sz[e] = a.z_fin[(size_t)bh * C::D + e];
    // padded rows of this range produce zeros
    for (int e = tid; e < (rend - max(r0, len)) * C::DV / 8; e += kThreadsTC)
        reinterpret_cast<uint4 *>(O + (size_t)max(r0, len) * C::DV)[e] = make_uint4(0, 0, 0, 0);
    fence_proxy_async_smem();
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tbase = *tslot;
    const uint32_t tmem_num = tbase + C::NU * NUS;

    if (warp == 8) {
        if (lane == 0 && ntiles > 0) {
            const uint32_t xa = smem_u32(Xb), pa = smem_u32(Pb), wa = smem_u32(Wop), sa = smem_u32(Sop);
            auto load_x = [&](int t) {
                const int x = t % NX;
                mbar_arrive_expect_tx(fullx + x, C::XT);
                for (int kb = 0; kb < C::KBX; ++kb)
                    tma_load_3d(Xb + x * C::XT + kb * 16384, &mapQ, kb * 64, r0 + t * 128, bh, fullx + x);
            };
            auto proj = [&](int t) {
                const int x = t % NX;
                issue_proj<C>(tbase + (t % NUS) * C::NU, xa + x * C::XT, wa);
                mma_commit(uready + (t % NUS));
                mma_commit(xfree + x);
            };
            bool failed = false;
            for (int t = 0; t < NX && t < ntiles; ++t) load_x(t);
            wait_or_fail(fullx, 0, failed, status);
            tc_fence_after();
            proj(0);
            for (int t = 0; t < ntiles && !failed; ++t) {
                const int p = t % NP, q = t % NN;
                if (t + 1 < ntiles) {
                    wait_or_fail(fullx + (t + 1) % NX, ((t + 1) / NX) & 1, failed, status);
                    tc_fence_after();
                    proj(t + 1);
                }
                if (t + NX < ntiles) {
                    wait_or_fail(xfree + t % NX, (t / NX) & 1, failed, status);
                    load_x(t + NX);
                }
                wait_or_fail(phiready + p, (t / NP) & 1, failed, status);
                if (t >= NN) wait_or_fail(numfree + q, ((t - NN) / NN) & 1, failed, status);
                tc_fence_after();
                constexpr uint32_t idN = idesc_bf16(128, 2 * C::DV, false, false);
                const uint32_t pt = pa + p * C::PT;
#pragma unroll
                for (int kb = 0; kb < C::NPB; ++kb)
#pragma unroll
                    for (int k = 0; k < 4; ++k)
                        mma_bf16_ss(tmem_num + q * 2 * C::DV, sdesc(pt + kb * 16384 + 32 * k, 16, 1024, kSwizzle128),
                                    sdesc(sa + kb * (2 * C::DV * 128) + 32 * k, 16, 1024, kSwizzle128), idN,
                                    (kb | k) != 0);
                mma_commit(numready + q);
                mma_commit(pfree + p);
            }
        }
    } else {
        const int h = warp >> 2, r = ((warp & 3) << 5) | lane;
        const uint32_t lrow = (uint32_t)((warp & 3) << 5) << 16;
        bool failed = false;
        for (int t = 0; t < ntiles; ++t) {
            const int p = t % NP, q = t % NN;
            const int row0 = r0 + t * 128;
            const int nvalid = min(128, r1 - row0);
            wait_or_fail(uready + t % NUS, (t / NUS) & 1, failed, status);
            if (t >= NP) wait_or_fail(pfree + p, ((t - NP) / NP) & 1, failed, status);
            tc_fence_after();
            uint8_t *pt = Pb + p * C::PT;
            const bool valid = r < nvalid;
            float den = 0.0f;
            const uint32_t ucol = tbase + lrow + (t % NUS) * C::NU;
            if (h == 0) phi_row_half<C, 0>(ucol, sT, sAB, sbias, valid, r, pt, nullptr, sz, den);
            else phi_row_half<C, 1>(ucol, sT, sAB, sbias, valid, r, pt, nullptr, sz, den);
            float *dslot = sden + (t & 1) * 256;
            dslot[h * 128 + r] = den;
            fence_proxy_async_smem();
            tc_fence_before();
            mbar_arrive(phiready + p);
            named_sync<kWorkers>(1);  // both halves of every row have written their part of the normaliser
            const float dsum = dslot[r] + dslot[128 + r] + a.eps;
            wait_or_fail(numready + q, (t / NN) & 1, failed, status);
            tc_fence_after();
            // this thread writes output columns [h*DV/2, (h+1)*DV/2) of row r
            constexpr int HC = C::DV / 2;
            uint4 outv[HC / 8];
#pragma unroll
            for (int c0 = 0; c0 < HC; c0 += 16) {
                uint32_t xh[16], xl[16];
                const uint32_t col = tmem_num + q * 2 * C::DV + h * HC + c0;
                tmem_ld16(lrow + col, xh);
                tmem_ld16(lrow + col + C::DV, xl);
                tmem_wait_ld();
                float o[16];
#pragma unroll
                for (int c = 0; c < 16; ++c)
                    o[c] = (dsum != 0.0f) ? (__uint_as_float(xh[c]) + __uint_as_float(xl[c])) / dsum : 0.0f;
#pragma unroll
                for (int c = 0; c < 16; c += 8)
                    outv[(c0 + c) / 8] = make_uint4(pack_bf16x2(o[c], o[c + 1]), pack_bf16x2(o[c + 2], o[c + 3]),
                                                    pack_bf16x2(o[c + 4], o[c + 5]), pack_bf16x2(o[c + 6], o[c + 7]));
            }
            tc_fence_before();
            mbar_arrive(numfree + q);
            if (valid) {
                uint4 *dst = reinterpret_cast<uint4 *>(O + (size_t)(row0 + r) * C::DV + h * HC);
#pragma unroll
                for (int k = 0; k < HC / 8; ++k) dst[k] = outv[k];
            }
        }
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 0) tmem_dealloc(tbase, C::TMEM_Q);
}

// ---------------------------------------------------------------------------
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

// (width, n, BH) bf16 tensor, boxes of 64 columns x 128 rows, 128B swizzle,
// out-of-range elements read as zero.
bool make_map(CUtensorMap *m, const void *base, int width, int n, int BH) {
    EncodeTiledFn enc = encoder();
    if (!enc) return false;
    cuuint64_t dims[3] = {(cuuint64_t)width, (cuuint64_t)n, (cuuint64_t)BH};
    cuuint64_t strides[2] = {(cuuint64_t)width * 2, (cuuint64_t)n * width * 2};
    cuuint32_t box[3] = {64, 128, 1};
    cuuint32_t es[3] = {1, 1, 1};
    return enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void *>(base), dims, strides, box, es,
               CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
               CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

int *status_word(const AttnArgs &a) { return reinterpret_cast<int *>(reinterpret_cast<char *>(a.counters) - 256); }

// The tensor-core kernels split each head into ranges of whole 128-row tiles
// (8 tiles by default; LUNA_TC_TILES_PER_SPLIT overrides it for tuning and for
// tests of long per-block tile loops).  There are never more ranges than the
// generic plan sized the workspace for.
AttnArgs tc_splits(const AttnArgs &a) {
    AttnArgs b = a;
    int tiles = 8;
    if (const char *env = getenv("LUNA_TC_TILES_PER_SPLIT")) {
        const int v = atoi(env);
        if (v > 0 && v < (1 << 20)) tiles = v;
    }
    const int ntile = (a.n + 127) / 128;
    if (tiles > ntile) tiles = ntile > 0 ? ntile : 1;
    while ((ntile + tiles - 1) / tiles > a.nsplit) ++tiles;
    b.rows_per_split = tiles * 128;
    b.nsplit = (a.n + b.rows_per_split - 1) / b.rows_per_split;
    return b;
}

template <class C>
cudaError_t fwd_tc(const AttnArgs &a0, cudaStream_t s) {
    const AttnArgs a = tc_splits(a0);
    CUtensorMap mK, mV, mQ;
    if (!make_map(&mK, a.K, a.d, a.n, a.B * a.H) || !make_map(&mV, a.V, a.dv, a.n, a.B * a.H) ||
        !make_map(&mQ, a.Q, a.d, a.n, a.B * a.H))
        return cudaErrorInvalidValue;
    cudaError_t e = cudaFuncSetAttribute(k_tc_keys<C>, cudaFuncAttributeMaxDynamicSharedMemorySize, C::SMEM_K);
    if (e != cudaSuccess) return e;
    e = cudaFuncSetAttribute(k_tc_query<C>, cudaFuncAttributeMaxDynamicSharedMemorySize, C::SMEM_Q);
    if (e != cudaSuccess) return e;
    int *st = status_word(a);
    LUNA_LAUNCH("tc_keys", k_tc_keys<C>, dim3(a.nsplit, a.B * a.H), kThreadsTC, C::SMEM_K, s, mK, mV, a, st);
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
    LUNA_LAUNCH("tc_query", k_tc_query<C>, dim3(a.nsplit, a.B * a.H), kThreadsTC, C::SMEM_Q, s, mQ, a, st);
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

TcPlan tc_plan(const luna_attn_desc &ad, const TableLayout &lay) {
    TcPlan p;
    p.variant = variant(ad, lay);
    p.eligible = p.variant >= 0 && encoder() != nullptr;
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

cudaError_t launch_tc_bwd(const TcPlan &, const AttnArgs &a, char *, bool have_stats, cudaStream_t s) {
    return launch_simt_bwd(a, LUNA_BF16, have_stats, s);
}

}  // namespace luna
