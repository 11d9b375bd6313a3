// One step of the streaming form (recurrent decode): for every (batch, head),
// with the state (S, z) after t tokens and the new token (q, k, v),
//     S <- S + phi(k) v^T,   z <- z + phi(k),   o = phi(q)^T S / (phi(q)^T z + eps)
// (the associative streaming form of Eq. kernel-attn named in the abstract and
// Sec. 3.2; the state after the token is the inclusive prefix of the causal form).
//
// One block per head.  The work per head is two projections of width d, 2*M
// interval searches and channel evaluations, and one pass over the D x dv
// fp32 state (read, update, write back) with the output accumulated on the
// way: the state traffic bounds the step, so it is CUDA-core code that reads
// and writes every state element once, in 16-byte accesses along the value
// columns.  The interval search block is staged in shared memory so that the searches do
// not wait on ten dependent global loads.
#include <math.h>

#include "luna_common.cuh"
#include "luna_prof.cuh"
#include "luna_simt.cuh"

namespace luna {

namespace {

constexpr int kDecThreads = 256;

template <typename IO> __device__ __forceinline__ float ld_io(const IO *p, int64_t i);
template <> __device__ __forceinline__ float ld_io<float>(const float *p, int64_t i) { return p[i]; }
template <> __device__ __forceinline__ float ld_io<__nv_bfloat16>(const __nv_bfloat16 *p, int64_t i) {
    return __bfloat162float(p[i]);
}
template <typename IO> __device__ __forceinline__ void st_io(IO *p, int64_t i, float v);
template <> __device__ __forceinline__ void st_io<float>(float *p, int64_t i, float v) { p[i] = v; }
template <> __device__ __forceinline__ void st_io<__nv_bfloat16>(__nv_bfloat16 *p, int64_t i, float v) {
    p[i] = __float2bfloat16_rn(v);
}

template <typename IO>
__global__ void __launch_bounds__(kDecThreads) k_decode(DecodeArgs a) {
    __shared__ float sx[2][kMaxD];        // q, k
    __shared__ float sv[kMaxD];
    __shared__ float sphi[2][kMaxFeat];   // phi(q), phi(k)
    __shared__ float su[2][32];           // projections of q and k
    __shared__ float so[4 * kDecThreads]; // output partials [feature group][column]
    __shared__ float sden[kDecThreads / 32];
    __shared__ __align__(16) float sTe[kEytzinger];
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int64_t bh = blockIdx.x;
    const int d = a.d, dv = a.dv, M = a.M, L = a.L, D = a.D;
    const char *table = a.table + (size_t)(bh % a.H) * a.table_stride;  // this head's table
    for (int e = tid; e < d; e += blockDim.x) {
        sx[0][e] = ld_io(static_cast<const IO *>(a.q), bh * d + e);
        sx[1][e] = ld_io(static_cast<const IO *>(a.k), bh * d + e);
    }
    for (int e = tid; e < dv; e += blockDim.x) sv[e] = ld_io(static_cast<const IO *>(a.v), bh * dv + e);
    const float4 *Te4 = reinterpret_cast<const float4 *>(table + a.lay.off_Te);
    for (int e = tid; e < kEytzinger / 4; e += blockDim.x) reinterpret_cast<float4 *>(sTe)[e] = __ldg(Te4 + e);
    __syncthreads();
    // u = W x + b for x = q, k: one warp per dot product
    const float *W = reinterpret_cast<const float *>(table + a.lay.off_W);
    const float *bias = reinterpret_cast<const float *>(table + a.lay.off_b);
    for (int p = warp; p < 2 * M; p += blockDim.x / 32) {
        const int side = p / M, m = p % M;
        float acc = 0.0f;
        for (int c = lane; c < d; c += 32) acc = fmaf(W[m * d + c], sx[side][c], acc);
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, o);
        if (lane == 0) su[side][m] = acc + bias[m];
    }
    __syncthreads();
    // phi: interval of u from the bucketed search block, then max(alpha u + beta, floor) per channel
    const float2 *AB = reinterpret_cast<const float2 *>(table + a.lay.off_AB);
    const float fl = channel_floor(a.lay);
    for (int p = tid; p < 2 * M; p += blockDim.x) {
        const int side = p / M, m = p % M;
        const float u = su[side][m];
        const int j = interval_bucketed(sTe, reinterpret_cast<const unsigned short *>(sTe + kSearchT), u);
        if (L == 8) {  // the (alpha, beta) of the 8 channels as four 16-byte loads in flight
            const float4 *ab4 = reinterpret_cast<const float4 *>(AB + (size_t)j * 8);
            float4 w[4];
#pragma unroll
            for (int k = 0; k < 4; ++k) w[k] = __ldg(ab4 + k);
#pragma unroll
            for (int k = 0; k < 4; ++k) {
                sphi[side][m * 8 + 2 * k] = fmaxf(fmaf(w[k].x, u, w[k].y), fl);
                sphi[side][m * 8 + 2 * k + 1] = fmaxf(fmaf(w[k].z, u, w[k].w), fl);
            }
        } else {
            for (int l = 0; l < L; ++l) {
                const float2 ab = __ldg(AB + (size_t)j * L + l);
                sphi[side][m * L + l] = fmaxf(fmaf(ab.x, u, ab.y), fl);
            }
        }
    }
    __syncthreads();
    // z <- z + phi(k); den = phi(q).z + eps
    float *z = a.z + bh * a.z_stride;
    float dp = 0.0f;
    for (int f = tid; f < D; f += blockDim.x) {
        const float zf = z[f] + sphi[1][f];
        z[f] = zf;
        dp = fmaf(sphi[0][f], zf, dp);
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) dp += __shfl_xor_sync(0xffffffffu, dp, o);
    if (lane == 0) sden[warp] = dp;
    // S <- S + phi(k) v^T and the numerator phi(q)^T S.  With dv % 4 == 0 and a 16-byte aligned state,
    // thread (g, c4) owns columns 4*c4 .. 4*c4+3 and features f = g (mod G); else one column per thread.
    float *S = a.S + bh * a.S_stride;
    const bool vec = (dv % 4 == 0) && ((reinterpret_cast<uintptr_t>(S) & 15) == 0) && (a.S_stride % 4 == 0);
    const int cw = vec ? dv / 4 : dv;  // column units per feature row
    const int G = kDecThreads / cw;    // feature groups (dv <= 128: G >= 2)
    const int g = tid / cw, cu = tid % cw;
    float num[4] = {0.0f, 0.0f, 0.0f, 0.0f};
    if (g < G) {
        if (vec) {
            const float4 vc = make_float4(sv[4 * cu], sv[4 * cu + 1], sv[4 * cu + 2], sv[4 * cu + 3]);
            float4 *S4 = reinterpret_cast<float4 *>(S);
            // R rows in flight: all loaded before any is stored (a store would otherwise order
            // the next load behind it, as the compiler cannot tell the rows apart)
            constexpr int R = 4;
            for (int f0 = g; f0 < D; f0 += R * G) {
                float4 sv4[R];
#pragma unroll
                for (int i = 0; i < R; ++i) {
                    const int f = f0 + i * G;
                    sv4[i] = f < D ? S4[(int64_t)f * cw + cu] : make_float4(0.f, 0.f, 0.f, 0.f);
                }
#pragma unroll
                for (int i = 0; i < R; ++i) {
                    const int f = f0 + i * G;
                    if (f < D) {
                        const float pk = sphi[1][f], pq = sphi[0][f];
                        float4 s = sv4[i];
                        s.x = fmaf(pk, vc.x, s.x); s.y = fmaf(pk, vc.y, s.y);
                        s.z = fmaf(pk, vc.z, s.z); s.w = fmaf(pk, vc.w, s.w);
                        S4[(int64_t)f * cw + cu] = s;
                        num[0] = fmaf(pq, s.x, num[0]); num[1] = fmaf(pq, s.y, num[1]);
                        num[2] = fmaf(pq, s.z, num[2]); num[3] = fmaf(pq, s.w, num[3]);
                    }
                }
            }
        } else {
            const float vc = sv[cu];
#pragma unroll 8
            for (int f = g; f < D; f += G) {
                const float s = fmaf(sphi[1][f], vc, S[(int64_t)f * dv + cu]);
                S[(int64_t)f * dv + cu] = s;
                num[0] = fmaf(sphi[0][f], s, num[0]);
            }
        }
    }
    if (g < G) {
        if (vec) {
#pragma unroll
            for (int e = 0; e < 4; ++e) so[g * dv + 4 * cu + e] = num[e];
        } else {
            so[g * dv + cu] = num[0];
        }
    }
    __syncthreads();
    if (tid < dv) {
        float den = a.eps;
        for (int w = 0; w < kDecThreads / 32; ++w) den += sden[w];
        float acc = 0.0f;
        for (int gg = 0; gg < G; ++gg) acc += so[gg * dv + tid];
        st_io(static_cast<IO *>(a.o), bh * dv + tid, den != 0.0f ? acc / den : 0.0f);
    }
}

}  // namespace

cudaError_t launch_decode(const DecodeArgs &a, luna_dtype io, cudaStream_t s) {
    if (a.BH == 0) return cudaSuccess;
    if (io == LUNA_F32)
        LUNA_LAUNCH("decode", k_decode<float>, a.BH, kDecThreads, 0, s, a);
    else
        LUNA_LAUNCH("decode", k_decode<__nv_bfloat16>, a.BH, kDecThreads, 0, s, a);
    return cudaGetLastError();
}

}  // namespace luna
