// C ABI of the LUNA library: argument checks, work planning, dispatch.
#include <math.h>
#include <string.h>

#include <algorithm>
#include <stdlib.h>

#include "luna_simt.cuh"
#include "luna_tc.cuh"

using namespace luna;

namespace {

constexpr size_t kMaxSmem = 227 * 1024;

int64_t cdiv(int64_t a, int64_t b) { return (a + b - 1) / b; }
int64_t round_up(int64_t a, int64_t b) { return cdiv(a, b) * b; }

luna_status check_phi(const luna_phi_desc *pd, int d) {
    if (!pd) return LUNA_ERR_INVALID_ARG;
    if (pd->M < 1 || pd->L < 1 || pd->hidden < 1 || d < 1) return LUNA_ERR_INVALID_ARG;
    if (pd->shared_channels != 0 && pd->shared_channels != 1) return LUNA_ERR_INVALID_ARG;
    if (pd->signed_outputs != 0 && pd->signed_outputs != 1) return LUNA_ERR_INVALID_ARG;
    if (!(pd->ch_rms_target >= 0.0f) || isinf(pd->ch_rms_target)) return LUNA_ERR_INVALID_ARG;
    if (pd->signed_outputs && pd->ch_rms_target > 0.0f) return LUNA_ERR_UNSUPPORTED;
    if (pd->param_head_stride < 0) return LUNA_ERR_INVALID_ARG;
    if (pd->param_head_stride) {  // one table per head, each a whole 256-byte aligned table
        const int64_t tb = table_layout(pd->M, pd->L, pd->hidden, d, pd->shared_channels).bytes;  // no variants here
        if (pd->param_head_stride < tb || pd->param_head_stride % 256 != 0) return LUNA_ERR_INVALID_ARG;
        if (pd->ch_rms_target > 0.0f) return LUNA_ERR_UNSUPPORTED;  // batch statistics of one shared map
    }
    if (pd->act < LUNA_ACT_RELU || pd->act > LUNA_ACT_TANH) return LUNA_ERR_INVALID_ARG;
    if ((pd->envelope != 0 && pd->envelope != 1) || (pd->bank_coef != 0 && pd->bank_coef != 1))
        return LUNA_ERR_INVALID_ARG;
    if ((pd->act || pd->envelope || pd->bank_coef) && (pd->ch_rms_target > 0.0f || pd->param_head_stride))
        return LUNA_ERR_UNSUPPORTED;
    if (pd->L > kMaxL || pd->M * pd->L > kMaxFeat || pd->M > 32 || pd->hidden > kMaxHidden ||
        pd->L * pd->hidden > kMaxUnits || d > kMaxD || pd->M * d > 4096)
        return LUNA_ERR_UNSUPPORTED;
    return LUNA_OK;
}

// Layout of the table of a descriptor (input width d).
TableLayout phi_layout(const luna_phi_desc *pd, int d) {
    return table_layout(pd->M, pd->L, pd->hidden, d, pd->shared_channels, pd->signed_outputs, pd->act, pd->envelope,
                        pd->bank_coef);
}

bool phi_variant(const luna_phi_desc *pd) { return pd->act || pd->envelope || pd->bank_coef; }

struct Plan {
    TableLayout lay;
    int BH = 0;
    int nsplit = 0, rps = 0, nsplit_b = 0, rps_b = 0;
    int seg_len = 0, nseg = 0;
    int gsize = 0;
    // workspace offsets (bytes)
    size_t o_counters = 0, o_status = 0, o_Spart = 0, o_zpart = 0, o_Sfin = 0, o_zfin = 0;
    size_t o_dSpart = 0, o_dzpart = 0, o_dSfin = 0, o_dzfin = 0, o_gpart = 0, o_hist = 0;
    size_t o_segS = 0, o_segz = 0, o_segdS = 0, o_segdz = 0, o_rowstat = 0;
    size_t o_dphi = 0, o_phik = 0, o_pq2 = 0;  // streaming-form backward on tensor cores
    size_t o_items = 0;                        // split of the tensor-core work items (non-causal)
    float ch_target = 0.0f;                    // channel RMS normalisation (non-causal; 0: off)
    size_t o_chpart = 0, o_chstat = 0, o_chsigma = 0, o_chkappa = 0, o_chT = 0;
    size_t o_chtab = 0;                        // streaming form: the sqrt(sigma)-scaled table
    size_t ws_fwd = 0, ws_bwd = 0, state_bytes = 0;
    TcPlan tc;
};

// Fixed state-segment length of the streaming form (tuning and tests: LUNA_CAUSAL_SEG_ROWS, a multiple of
// 128 rows).  The segment length decides the layout of the forward state that luna_attn_bwd,
// luna_state_final and luna_attn_decode read back, so the variable is read once, when the library is
// loaded, and every call of the process plans with the same value.
int read_seg_rows_override() {
    const char *env = getenv("LUNA_CAUSAL_SEG_ROWS");
    if (!env) return 0;
    const long v = atol(env);
    return (v >= 128 && v % 128 == 0 && v < (1L << 24)) ? (int)v : 0;
}
const int g_seg_rows_override = read_seg_rows_override();

struct Bump {
    size_t n = 0;
    size_t take(size_t bytes) {
        size_t o = n;
        n += (bytes + 255) & ~size_t(255);
        return o;
    }
};

luna_status make_plan(const luna_attn_desc *ad, const luna_phi_desc *pd, Plan &p) {
    if (!ad) return LUNA_ERR_INVALID_ARG;
    if (ad->B < 0 || ad->H < 0 || ad->n < 0 || ad->d < 1 || ad->dv < 1) return LUNA_ERR_INVALID_ARG;
    if (ad->io != LUNA_F32 && ad->io != LUNA_BF16) return LUNA_ERR_INVALID_ARG;
    if (ad->causal != 0 && ad->causal != 1) return LUNA_ERR_INVALID_ARG;
    if (!(ad->eps >= 0.0f) || isinf(ad->eps)) return LUNA_ERR_INVALID_ARG;
    if (ad->chunk != 0 && (ad->chunk < 16 || ad->chunk > 128 || ad->chunk % 16 != 0)) return LUNA_ERR_INVALID_ARG;
    luna_status st = check_phi(pd, ad->d);
    if (st != LUNA_OK) return st;
    if (ad->dv > kMaxD || ad->n > (1 << 24)) return LUNA_ERR_UNSUPPORTED;
    p.ch_target = pd->ch_rms_target;
    if ((int64_t)ad->B * ad->H > (1 << 24)) return LUNA_ERR_UNSUPPORTED;

    p.lay = phi_layout(pd, ad->d);
    const int BH = ad->B * ad->H, n = ad->n, D = p.lay.D, dv = ad->dv;
    p.BH = BH;
    p.gsize = grad_words(p.lay);
    if (BH == 0 || n == 0) return LUNA_OK;
    // splits depend only on the descriptor, so workspace sizes are reproducible
    {
        int64_t target = std::max<int64_t>(1, cdiv(1216, BH));
        int64_t ns = std::min<int64_t>(target, cdiv(n, 32));
        p.rps = (int)round_up(cdiv(n, ns), 32);
        p.nsplit = (int)cdiv(n, p.rps);
        int64_t tb = std::max<int64_t>(1, cdiv(608, BH));
        int64_t nb = std::min<int64_t>(tb, cdiv(n, 16));
        p.rps_b = (int)round_up(cdiv(n, nb), 16);
        p.nsplit_b = (int)cdiv(n, p.rps_b);
        int64_t nc = std::min<int64_t>(std::min<int64_t>(target, 64), cdiv(n, 16));
        p.seg_len = (int)round_up(cdiv(n, nc), 128);  // whole 128-row tiles (tensor-core streaming form)
        if (g_seg_rows_override > 0) p.seg_len = g_seg_rows_override;
        p.nseg = (int)cdiv(n, p.seg_len);
    }
    const size_t f = sizeof(float);
    const size_t SD = (size_t)D * dv;
    Bump w;
    p.o_status = w.take(sizeof(int));  // offset 0: device status word of the last call
    p.o_counters = w.take(2 * (size_t)BH * sizeof(int));
    if (!ad->causal) {
        p.o_Spart = w.take((size_t)BH * p.nsplit * SD * f);
        p.o_zpart = w.take((size_t)BH * p.nsplit * D * f);
        p.o_Sfin = w.take((size_t)BH * SD * f);
        p.o_zfin = w.take((size_t)BH * D * f);
        p.o_items = w.take((kMaxGrid + 1 + 2 * (size_t)BH) * sizeof(int));
        if (p.ch_target > 0.0f) {
            p.o_chpart = w.take(2 * (size_t)kChStatBlocks * p.lay.L * f);
            p.o_chstat = w.take(8 * (size_t)kMaxL * sizeof(double));
            p.o_chsigma = w.take((size_t)kMaxL * f);
            p.o_chkappa = w.take(2 * (size_t)kMaxL * f);
            p.o_chT = w.take((size_t)BH * p.lay.L * sizeof(double));
        }
        p.ws_fwd = w.n;
        // per-head partial slots: generic splits, or (tensor-core path) runs of work items, never more
        // than the forward split count
        const size_t nslot = (size_t)std::max(p.nsplit, p.nsplit_b);
        p.o_dSpart = w.take((size_t)BH * nslot * SD * f);
        p.o_dzpart = w.take((size_t)BH * nslot * D * f);
        p.o_dSfin = w.take((size_t)BH * SD * f);
        p.o_dzfin = w.take((size_t)BH * D * f);
        // with channel normalisation, the partials of the scale term of the backward follow
        // parameter-gradient partials: fp32 (tensor-core kernels) or fp64 (generic kernels)
        p.o_gpart = w.take((2 * (size_t)BH * p.nsplit_b + (p.ch_target > 0.0f ? 2 * kChKBlocks : 0)) * p.gsize *
                           sizeof(double));
        p.o_hist = w.take((size_t)p.gsize * sizeof(double));
        p.ws_bwd = w.n;
        p.state_bytes = (size_t)BH * (SD + D) * f;
    } else {
        const int ns = p.nseg;
        p.o_Spart = w.take((size_t)BH * ns * SD * f);
        p.o_zpart = w.take((size_t)BH * ns * D * f);
        p.o_segS = w.take((size_t)BH * (ns + 1) * SD * f);
        p.o_segz = w.take((size_t)BH * (ns + 1) * D * f);
        if (p.ch_target > 0.0f) {
            p.o_chpart = w.take(2 * (size_t)kChStatBlocks * p.lay.L * f);
            p.o_chstat = w.take(8 * (size_t)kMaxL * sizeof(double));
            p.o_chsigma = w.take((size_t)kMaxL * f);
            p.o_chkappa = w.take(2 * (size_t)kMaxL * f);
            // T rows: one per block of the tensor-core chain rule or per (head, segment) of the generic one
            p.o_chT = w.take((size_t)std::max<int64_t>(kMaxGrid, (int64_t)BH * ns) * p.lay.L * sizeof(double));
            p.o_chtab = w.take((size_t)p.lay.bytes);
        }
        p.ws_fwd = w.n;
        p.o_dSpart = w.take((size_t)BH * ns * SD * f);
        p.o_dzpart = w.take((size_t)BH * ns * D * f);
        p.o_segdS = w.take((size_t)BH * ns * SD * f);
        p.o_segdz = w.take((size_t)BH * ns * D * f);
        p.o_rowstat = w.take((size_t)BH * n * 2 * f);
        p.o_gpart = w.take((2 * (size_t)BH * ns + (p.ch_target > 0.0f ? 2 * kChKBlocks : 0)) * p.gsize *
                           sizeof(double));
        p.o_hist = w.take((size_t)p.gsize * sizeof(double));
        p.ws_bwd = w.n;
        p.state_bytes = (size_t)BH * (ns + 1) * (SD + D) * f;
    }
    p.tc = tc_plan(*ad, p.lay);
    if (p.tc.eligible) {
        p.ws_fwd = std::max(p.ws_fwd, p.tc.ws_fwd);
        p.ws_bwd = std::max(p.ws_bwd, p.tc.ws_bwd);
    }
    if (ad->causal && p.tc.causal_bwd) {  // dphi (fp32), phi(k) and phi(q)/den as hi|lo (bf16) of every row
        Bump wb;
        wb.n = p.ws_bwd;
        const size_t R = (size_t)BH * n;
        p.o_dphi = wb.take(R * D * f);
        p.o_phik = wb.take(R * 2 * D * 2);
        p.o_pq2 = wb.take(R * 2 * D * 2);
        p.ws_bwd = wb.n;
    }
    return LUNA_OK;
}

AttnArgs make_args(const luna_attn_desc *ad, const Plan &p, const void *table, const void *Q, const void *K,
                   const void *V, const int32_t *lengths, void *ws) {
    AttnArgs a;
    memset(&a, 0, sizeof(a));
    a.B = ad->B; a.H = ad->H; a.n = ad->n; a.d = ad->d; a.dv = ad->dv;
    a.M = p.lay.M; a.L = p.lay.L; a.D = p.lay.D;
    a.eps = ad->eps;
    a.lay = p.lay;
    a.hs_mul = 1;
    a.table = static_cast<const char *>(table);
    a.Q = Q; a.K = K; a.V = V;
    a.lengths = lengths;
    char *w = static_cast<char *>(ws);
    a.counters = reinterpret_cast<int *>(w + p.o_counters);
    a.nsplit = p.nsplit; a.rows_per_split = p.rps;
    a.nsplit_b = p.nsplit_b; a.rows_per_split_b = p.rps_b;
    a.gsize = p.gsize;
    a.chunk = ad->chunk ? ad->chunk : 64;
    a.seg_len = p.seg_len; a.nseg = p.nseg;
    a.S_part = reinterpret_cast<float *>(w + p.o_Spart);
    a.z_part = reinterpret_cast<float *>(w + p.o_zpart);
    if (!ad->causal) {
        a.S_fin = reinterpret_cast<float *>(w + p.o_Sfin);
        a.z_fin = reinterpret_cast<float *>(w + p.o_zfin);
        a.items_ws = reinterpret_cast<int *>(w + p.o_items);
        if (p.ch_target > 0.0f) {
            a.ch_target = p.ch_target;
            a.ch_io = ad->io;
            a.ch_part = reinterpret_cast<float *>(w + p.o_chpart);
            a.ch_stat = reinterpret_cast<double *>(w + p.o_chstat);
            a.ch_sigma = reinterpret_cast<float *>(w + p.o_chsigma);
            a.ch_kappa = reinterpret_cast<float *>(w + p.o_chkappa);
            a.ch_T = reinterpret_cast<double *>(w + p.o_chT);
        }
    } else {
        a.seg_S = reinterpret_cast<float *>(w + p.o_segS);
        a.seg_z = reinterpret_cast<float *>(w + p.o_segz);
        if (p.ch_target > 0.0f) {
            a.ch_target = p.ch_target;
            a.ch_io = ad->io;
            a.ch_causal = 1;
            a.ch_part = reinterpret_cast<float *>(w + p.o_chpart);
            a.ch_stat = reinterpret_cast<double *>(w + p.o_chstat);
            a.ch_sigma = reinterpret_cast<float *>(w + p.o_chsigma);
            a.ch_kappa = reinterpret_cast<float *>(w + p.o_chkappa);
            a.ch_T = reinterpret_cast<double *>(w + p.o_chT);
        }
    }
    return a;
}

void point_state(const luna_attn_desc *ad, const Plan &p, AttnArgs &a, void *state) {
    if (!state) return;
    float *s = static_cast<float *>(state);
    const size_t SD = (size_t)p.lay.D * ad->dv;
    if (!ad->causal) {
        a.S_fin = s;
        a.z_fin = s + (size_t)p.BH * SD;
    } else {
        a.seg_S = s;
        a.seg_z = s + (size_t)p.BH * (p.nseg + 1) * SD;
    }
}

luna_status cuda_status(cudaError_t e) { return e == cudaSuccess ? LUNA_OK : LUNA_ERR_CUDA; }

// Per-head parameters: the sub-problem of head index h of every sequence.  Its B heads are the caller's
// heads (b, h): the tensors start at head h and step H heads (hs_mul = H), the state and the gradients
// start at head h's block, and the table is head h's.  Workspace buffers are indexed by the sub-problem's
// own head numbers, so the sub-problems run one after another on the stream.
AttnArgs head_args(const AttnArgs &a, const luna_attn_desc *ad, const luna_phi_desc *pd, const Plan &p, int h) {
    AttnArgs s = a;
    const size_t eb = ad->io == LUNA_F32 ? 4 : 2;
    const size_t oq = (size_t)h * ad->n * ad->d * eb, ov = (size_t)h * ad->n * ad->dv * eb;
    auto at = [](const void *x, size_t o) -> const void * {
        return x ? static_cast<const void *>(static_cast<const char *>(x) + o) : nullptr;
    };
    auto atw = [](void *x, size_t o) -> void * { return x ? static_cast<void *>(static_cast<char *>(x) + o) : nullptr; };
    s.Q = at(a.Q, oq); s.K = at(a.K, oq); s.V = at(a.V, ov); s.dO = at(a.dO, ov);
    s.O = atw(a.O, ov); s.dQ = atw(a.dQ, oq); s.dK = atw(a.dK, oq); s.dV = atw(a.dV, ov);
    s.H = 1;
    s.hs_mul = ad->H;
    s.table = a.table + (size_t)h * pd->param_head_stride;
    const size_t D = p.lay.D, SD = D * ad->dv;
    if (!ad->causal) {
        s.S_fin = a.S_fin + (size_t)h * SD;
        s.z_fin = a.z_fin + (size_t)h * D;
    } else {
        s.seg_S = a.seg_S + (size_t)h * (p.nseg + 1) * SD;
        s.seg_z = a.seg_z + (size_t)h * (p.nseg + 1) * D;
    }
    const size_t Md = (size_t)pd->M * ad->d, fc1 = pd->shared_channels ? pd->hidden : (size_t)pd->L * pd->hidden;
    if (s.grads.dW) {
        s.grads.dW += h * Md; s.grads.db += (size_t)h * pd->M;
        s.grads.dw1 += h * fc1; s.grads.db1 += h * fc1;
        s.grads.dw2 += (size_t)h * pd->L * pd->hidden; s.grads.db2 += (size_t)h * pd->L;
    }
    return s;
}

bool aligned(const void *p, size_t a) { return (reinterpret_cast<uintptr_t>(p) % a) == 0; }

}  // namespace

extern "C" {

int luna_version(void) { return 100; }

const char *luna_status_string(luna_status s) {
    switch (s) {
        case LUNA_OK: return "LUNA_OK";
        case LUNA_ERR_INVALID_ARG: return "LUNA_ERR_INVALID_ARG";
        case LUNA_ERR_UNSUPPORTED: return "LUNA_ERR_UNSUPPORTED";
        case LUNA_ERR_WORKSPACE: return "LUNA_ERR_WORKSPACE";
        case LUNA_ERR_CUDA: return "LUNA_ERR_CUDA";
        case LUNA_ERR_DEVICE_TIMEOUT: return "LUNA_ERR_DEVICE_TIMEOUT";
    }
    return "LUNA_ERR_UNKNOWN";
}

luna_status luna_phi_table_size(const luna_phi_desc *pd, int d, size_t *bytes) {
    if (!bytes) return LUNA_ERR_INVALID_ARG;
    luna_status st = check_phi(pd, d);
    if (st != LUNA_OK) return st;
    *bytes = (size_t)phi_layout(pd, d).bytes;
    return LUNA_OK;
}

luna_status luna_phi_prepare(const luna_phi_desc *pd, int d, const luna_phi_params *params, void *table,
                             size_t table_bytes, void *stream) {
    luna_status st = check_phi(pd, d);
    if (st != LUNA_OK) return st;
    if (!params || !table || !params->W || !params->b || !params->w1 || !params->b1 || !params->w2 || !params->b2)
        return LUNA_ERR_INVALID_ARG;
    if ((pd->envelope && (!params->We || !params->be)) || (pd->bank_coef && !params->coef)) return LUNA_ERR_INVALID_ARG;
    if (!aligned(table, 256)) return LUNA_ERR_INVALID_ARG;
    TableLayout lay = phi_layout(pd, d);
    if (table_bytes < (size_t)lay.bytes) return LUNA_ERR_WORKSPACE;
    return cuda_status(launch_phi_prepare(*params, lay, table, static_cast<cudaStream_t>(stream)));
}

luna_status luna_featmap(const luna_phi_desc *pd, int d, const void *table, const void *X, luna_dtype xtype,
                         int64_t rows, float *Phi, void *stream) {
    luna_status st = check_phi(pd, d);
    if (st != LUNA_OK) return st;
    if (rows < 0 || (xtype != LUNA_F32 && xtype != LUNA_BF16)) return LUNA_ERR_INVALID_ARG;
    if (pd->ch_rms_target > 0.0f) return LUNA_ERR_UNSUPPORTED;
    if (pd->param_head_stride) return LUNA_ERR_UNSUPPORTED;  // rows carry no head: pass that head's table
    if (rows == 0) return LUNA_OK;
    if (!table || !X || !Phi) return LUNA_ERR_INVALID_ARG;
    TableLayout lay = phi_layout(pd, d);
    return cuda_status(launch_featmap(lay, static_cast<const char *>(table), X, xtype, rows, Phi,
                                      static_cast<cudaStream_t>(stream)));
}

luna_status luna_workspace_size(const luna_attn_desc *ad, const luna_phi_desc *pd, int backward, size_t *bytes) {
    if (!bytes) return LUNA_ERR_INVALID_ARG;
    Plan p;
    luna_status st = make_plan(ad, pd, p);
    if (st != LUNA_OK) return st;
    *bytes = backward ? p.ws_bwd : p.ws_fwd;
    if (*bytes == 0) *bytes = 256;
    return LUNA_OK;
}

luna_status luna_state_size(const luna_attn_desc *ad, const luna_phi_desc *pd, size_t *bytes) {
    if (!bytes) return LUNA_ERR_INVALID_ARG;
    Plan p;
    luna_status st = make_plan(ad, pd, p);
    if (st != LUNA_OK) return st;
    *bytes = p.state_bytes ? p.state_bytes : 256;
    return LUNA_OK;
}

luna_status luna_attn_fwd(const luna_attn_desc *ad, const luna_phi_desc *pd, const void *table, const void *Q,
                          const void *K, const void *V, const int32_t *lengths, void *O, void *state,
                          void *workspace, size_t ws_bytes, void *stream) {
    Plan p;
    luna_status st = make_plan(ad, pd, p);
    if (st != LUNA_OK) return st;
    if (p.BH == 0 || ad->n == 0) return LUNA_OK;
    if (!table || !Q || !K || !V || !O || !workspace) return LUNA_ERR_INVALID_ARG;
    if (!aligned(workspace, 256) || !aligned(table, 256) || (state && !aligned(state, 256)))
        return LUNA_ERR_INVALID_ARG;
    if (ws_bytes < p.ws_fwd) return LUNA_ERR_WORKSPACE;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    AttnArgs a = make_args(ad, p, table, Q, K, V, lengths, workspace);
    a.O = O;
    point_state(ad, p, a, state);
    if ((!ad->causal ? simt_max_smem(a) : causal_max_smem(a)) > kMaxSmem && !p.tc.eligible)
        return LUNA_ERR_UNSUPPORTED;
    if (a.ch_sigma && chrms_max_smem(a) > kMaxSmem) return LUNA_ERR_UNSUPPORTED;
    cudaError_t e = cudaMemsetAsync(workspace, 0, p.o_counters + 2 * sizeof(int) * (size_t)p.BH, s);
    if (e != cudaSuccess) return LUNA_ERR_CUDA;
    if (a.ch_sigma && (e = launch_chrms_stats(a, ad->io, s)) != cudaSuccess) return LUNA_ERR_CUDA;
    if (a.ch_causal) {  // the streaming form runs on the sqrt(sigma)-scaled table
        if ((e = launch_chrms_table(a, static_cast<char *>(workspace) + p.o_chtab, s)) != cudaSuccess)
            return LUNA_ERR_CUDA;
        a.table = static_cast<const char *>(workspace) + p.o_chtab;
    }
    const int nsub = pd->param_head_stride ? ad->H : 1;  // per-head parameters: one sub-problem per head index
    for (int h = 0; h < nsub; ++h) {
        const AttnArgs b = pd->param_head_stride ? head_args(a, ad, pd, p, h) : a;
        if (ad->causal) {
            if (p.tc.causal_fwd && tc_inputs_ok(TcPlan{true}, b.Q, b.K, b.V, b.O)) e = launch_tc_causal_fwd(b, s);
            else e = launch_causal_fwd(b, ad->io, state != nullptr, s);
        } else if (p.tc.eligible && tc_inputs_ok(p.tc, b.Q, b.K, b.V, b.O)) {
            e = launch_tc_fwd(p.tc, b, static_cast<char *>(workspace), s);
        } else {
            e = launch_simt_fwd(b, ad->io, s);
        }
        if (e != cudaSuccess) return LUNA_ERR_CUDA;
    }
    return LUNA_OK;
}

luna_status luna_attn_bwd(const luna_attn_desc *ad, const luna_phi_desc *pd, const void *table, const void *Q,
                          const void *K, const void *V, const void *dO, const int32_t *lengths, const void *state,
                          void *dQ, void *dK, void *dV, const luna_phi_grads *grads, void *workspace,
                          size_t ws_bytes, void *stream) {
    Plan p;
    luna_status st = make_plan(ad, pd, p);
    if (st != LUNA_OK) return st;
    if (!grads || !grads->dW || !grads->db || !grads->dw1 || !grads->db1 || !grads->dw2 || !grads->db2)
        return LUNA_ERR_INVALID_ARG;
    if ((pd->envelope && (!grads->dWe || !grads->dbe)) || (pd->bank_coef && !grads->dcoef)) return LUNA_ERR_INVALID_ARG;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    if (p.BH == 0 || ad->n == 0) {  // empty problem: parameter gradients are zero
        const size_t G = pd->param_head_stride ? (size_t)ad->H : 1;  // parameter sets
        const size_t Md = G * pd->M * ad->d, P = G * pd->L * pd->hidden;
        const size_t P1 = pd->shared_channels ? G * pd->hidden : P;  // fc1 entries
        cudaError_t e = cudaMemsetAsync(grads->dW, 0, Md * 4, s);
        if (e == cudaSuccess) e = cudaMemsetAsync(grads->db, 0, G * pd->M * 4, s);
        if (e == cudaSuccess) e = cudaMemsetAsync(grads->dw1, 0, P1 * 4, s);
        if (e == cudaSuccess) e = cudaMemsetAsync(grads->db1, 0, P1 * 4, s);
        if (e == cudaSuccess) e = cudaMemsetAsync(grads->dw2, 0, P * 4, s);
        if (e == cudaSuccess) e = cudaMemsetAsync(grads->db2, 0, G * pd->L * 4, s);
        if (e == cudaSuccess && pd->envelope) e = cudaMemsetAsync(grads->dWe, 0, (size_t)pd->L * ad->d * 4, s);
        if (e == cudaSuccess && pd->envelope) e = cudaMemsetAsync(grads->dbe, 0, (size_t)pd->L * 4, s);
        if (e == cudaSuccess && pd->bank_coef) e = cudaMemsetAsync(grads->dcoef, 0, (size_t)pd->L * 4, s);
        return cuda_status(e);
    }
    if (!table || !Q || !K || !V || !dO || !dQ || !dK || !dV || !workspace) return LUNA_ERR_INVALID_ARG;
    if (!aligned(workspace, 256) || !aligned(table, 256) || (state && !aligned(state, 256)))
        return LUNA_ERR_INVALID_ARG;
    if (ws_bytes < p.ws_bwd) return LUNA_ERR_WORKSPACE;
    AttnArgs a = make_args(ad, p, table, Q, K, V, lengths, workspace);
    char *w = static_cast<char *>(workspace);
    a.dO = dO; a.dQ = dQ; a.dK = dK; a.dV = dV;
    a.grads = *grads;
    a.dS_part = reinterpret_cast<float *>(w + p.o_dSpart);
    a.dz_part = reinterpret_cast<float *>(w + p.o_dzpart);
    a.gpart = reinterpret_cast<float *>(w + p.o_gpart);
    a.hist = reinterpret_cast<double *>(w + p.o_hist);
    if (!ad->causal) {
        a.dS_fin = reinterpret_cast<float *>(w + p.o_dSfin);
        a.dz_fin = reinterpret_cast<float *>(w + p.o_dzfin);
    } else {
        a.seg_dS = reinterpret_cast<float *>(w + p.o_segdS);
        a.seg_dz = reinterpret_cast<float *>(w + p.o_segdz);
        a.rowstat = reinterpret_cast<float *>(w + p.o_rowstat);
    }
    point_state(ad, p, a, const_cast<void *>(state));
    if ((!ad->causal ? simt_max_smem(a) : causal_max_smem(a)) > kMaxSmem && !p.tc.eligible)
        return LUNA_ERR_UNSUPPORTED;
    if (a.ch_sigma && chrms_max_smem(a) > kMaxSmem) return LUNA_ERR_UNSUPPORTED;
    cudaError_t e = cudaMemsetAsync(workspace, 0, p.o_counters + 2 * sizeof(int) * (size_t)p.BH, s);
    if (e != cudaSuccess) return LUNA_ERR_CUDA;
    if (a.ch_sigma && (e = launch_chrms_stats(a, ad->io, s)) != cudaSuccess) return LUNA_ERR_CUDA;
    if (a.ch_causal) {  // the streaming form runs on the sqrt(sigma)-scaled table
        if ((e = launch_chrms_table(a, w + p.o_chtab, s)) != cudaSuccess) return LUNA_ERR_CUDA;
        a.table = w + p.o_chtab;
    }
    if (ad->causal && p.tc.causal_bwd) {
        a.dphi = reinterpret_cast<float *>(w + p.o_dphi);
        a.phik = w + p.o_phik;
        a.pq2 = w + p.o_pq2;
    }
    const int nsub = pd->param_head_stride ? ad->H : 1;  // per-head parameters: one sub-problem per head index
    for (int h = 0; h < nsub; ++h) {
        const AttnArgs b = pd->param_head_stride ? head_args(a, ad, pd, p, h) : a;
        if (ad->causal) {
            if (p.tc.causal_bwd && tc_inputs_ok(TcPlan{true}, b.Q, b.K, b.V, b.dO) &&
                tc_inputs_ok(TcPlan{true}, b.dQ, b.dK, b.dV, nullptr))
                e = launch_tc_causal_bwd(b, state != nullptr, s);
            else
                e = launch_causal_bwd(b, ad->io, state != nullptr, s);
        } else if (p.tc.eligible && tc_inputs_ok(p.tc, b.Q, b.K, b.V, b.dO) &&
                   tc_inputs_ok(p.tc, b.dQ, b.dK, b.dV, nullptr)) {
            e = launch_tc_bwd(p.tc, b, w, state != nullptr, s);
        } else {
            e = launch_simt_bwd(b, ad->io, state != nullptr, s);
        }
        if (e != cudaSuccess) return LUNA_ERR_CUDA;
    }
    return LUNA_OK;
}

luna_status luna_attn_weights(const luna_attn_desc *ad, const luna_phi_desc *pd, const void *table, const void *Q,
                              const void *K, const int32_t *lengths, int row0, int rows, int teacher, float *A,
                              void *stream) {
    if (!ad) return LUNA_ERR_INVALID_ARG;
    if (ad->B < 0 || ad->H < 0 || ad->n < 0 || ad->d < 1 || ad->dv < 1) return LUNA_ERR_INVALID_ARG;
    if (ad->io != LUNA_F32 && ad->io != LUNA_BF16) return LUNA_ERR_INVALID_ARG;
    if (ad->causal != 0 && ad->causal != 1) return LUNA_ERR_INVALID_ARG;
    if (!(ad->eps >= 0.0f) || isinf(ad->eps)) return LUNA_ERR_INVALID_ARG;
    if (teacher != 0 && teacher != 1) return LUNA_ERR_INVALID_ARG;
    if (row0 < 0 || rows < 0 || (int64_t)row0 + rows > ad->n) return LUNA_ERR_INVALID_ARG;
    luna_status st = check_phi(pd, ad->d);
    if (st != LUNA_OK) return st;
    if (pd->ch_rms_target > 0.0f) return LUNA_ERR_UNSUPPORTED;  // batch statistics: not for a block of rows
    if (phi_variant(pd)) return LUNA_ERR_UNSUPPORTED;
    if (ad->n > (1 << 24) || (int64_t)ad->B * ad->H > 65535) return LUNA_ERR_UNSUPPORTED;
    if ((int64_t)ad->B * ad->H == 0 || rows == 0 || ad->n == 0) return LUNA_OK;
    if (!Q || !K || !A || (!teacher && !table)) return LUNA_ERR_INVALID_ARG;
    if (table && !aligned(table, 256)) return LUNA_ERR_INVALID_ARG;
    AttnArgs a;
    memset(&a, 0, sizeof(a));
    a.B = ad->B; a.H = ad->H; a.n = ad->n; a.d = ad->d; a.dv = ad->dv;
    a.lay = phi_layout(pd, ad->d);
    a.M = a.lay.M; a.L = a.lay.L; a.D = a.lay.D;
    a.eps = ad->eps;
    a.table = static_cast<const char *>(table);
    a.Q = Q; a.K = K;
    a.lengths = lengths;
    if (weights_max_smem(a) > kMaxSmem) return LUNA_ERR_UNSUPPORTED;
    return cuda_status(launch_weights(a, ad->io, ad->causal, row0, rows, teacher, pd->param_head_stride, A,
                                      static_cast<cudaStream_t>(stream)));
}

luna_status luna_state_final(const luna_attn_desc *ad, const luna_phi_desc *pd, void *state, float **S,
                             int64_t *S_stride, float **z, int64_t *z_stride) {
    if (!S || !S_stride || !z || !z_stride) return LUNA_ERR_INVALID_ARG;
    Plan p;
    luna_status st = make_plan(ad, pd, p);
    if (st != LUNA_OK) return st;
    if (!ad->causal) return LUNA_ERR_INVALID_ARG;
    if (!state) return LUNA_ERR_INVALID_ARG;
    const int64_t SD = (int64_t)p.lay.D * ad->dv, ns = p.nseg;
    float *base = static_cast<float *>(state);
    *S = base + ns * SD;  // segment prefixes [BH][nseg + 1][D][dv]: entry nseg is the total
    *S_stride = (ns + 1) * SD;
    *z = base + (int64_t)p.BH * (ns + 1) * SD + ns * p.lay.D;
    *z_stride = (ns + 1) * p.lay.D;
    return LUNA_OK;
}

luna_status luna_attn_decode(const luna_attn_desc *ad, const luna_phi_desc *pd, const void *table, const void *q,
                             const void *k, const void *v, void *o, float *S, int64_t S_stride, float *z,
                             int64_t z_stride, void *stream) {
    if (!ad) return LUNA_ERR_INVALID_ARG;
    if (ad->B < 0 || ad->H < 0 || ad->d < 1 || ad->dv < 1) return LUNA_ERR_INVALID_ARG;
    if (ad->io != LUNA_F32 && ad->io != LUNA_BF16) return LUNA_ERR_INVALID_ARG;
    if (!(ad->eps >= 0.0f) || isinf(ad->eps)) return LUNA_ERR_INVALID_ARG;
    luna_status st = check_phi(pd, ad->d);
    if (st != LUNA_OK) return st;
    if (ad->dv > kMaxD) return LUNA_ERR_UNSUPPORTED;
    if (pd->ch_rms_target > 0.0f) return LUNA_ERR_UNSUPPORTED;  // a batch statistic: no single-token step
    if (phi_variant(pd)) return LUNA_ERR_UNSUPPORTED;
    const int64_t BH = (int64_t)ad->B * ad->H;
    if (BH > (1 << 24)) return LUNA_ERR_UNSUPPORTED;
    const TableLayout lay = phi_layout(pd, ad->d);
    const int64_t SD = (int64_t)lay.D * ad->dv;
    if (S_stride == 0) S_stride = SD;
    if (z_stride == 0) z_stride = lay.D;
    if (S_stride < SD || z_stride < lay.D) return LUNA_ERR_INVALID_ARG;
    if (BH == 0) return LUNA_OK;
    if (!table || !q || !k || !v || !o || !S || !z) return LUNA_ERR_INVALID_ARG;
    if (!aligned(table, 256)) return LUNA_ERR_INVALID_ARG;
    DecodeArgs a;
    a.BH = (int)BH; a.d = ad->d; a.dv = ad->dv; a.M = lay.M; a.L = lay.L; a.D = lay.D;
    a.eps = ad->eps;
    a.lay = lay;
    a.table = static_cast<const char *>(table);
    a.H = ad->H;
    a.table_stride = pd->param_head_stride;
    a.q = q; a.k = k; a.v = v; a.o = o;
    a.S = S; a.z = z;
    a.S_stride = S_stride; a.z_stride = z_stride;
    return cuda_status(launch_decode(a, ad->io, static_cast<cudaStream_t>(stream)));
}

luna_status luna_selftest_wait(void *workspace, int64_t limit_ns, void *stream) {
    if (!workspace || !aligned(workspace, 256) || limit_ns <= 0 || limit_ns > 1000000000LL)
        return LUNA_ERR_INVALID_ARG;
    return cuda_status(launch_selftest_wait(static_cast<int *>(workspace), (long long)limit_ns,
                                            static_cast<cudaStream_t>(stream)));
}

luna_status luna_device_status(void *workspace, void *stream) {
    if (!workspace) return LUNA_ERR_INVALID_ARG;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    int word = 0;
    cudaError_t e = cudaMemcpyAsync(&word, workspace, sizeof(int), cudaMemcpyDeviceToHost, s);
    if (e == cudaSuccess) e = cudaStreamSynchronize(s);
    if (e == cudaSuccess && word != 0) e = cudaMemsetAsync(workspace, 0, sizeof(int), s);
    if (e == cudaSuccess) e = cudaStreamSynchronize(s);
    if (e != cudaSuccess) return LUNA_ERR_CUDA;
    return word == 0 ? LUNA_OK : LUNA_ERR_DEVICE_TIMEOUT;
}

}  // extern "C"
