/*
 * LUNA oracle: a plain, slow fp64 CPU restatement of the method.
 *
 * TEST INFRASTRUCTURE ONLY.  Nothing in the library path may call, link or
 * execute this file; only the tests, the graft smoke check and the CPU
 * baseline leg of the benchmark use it.  It shares no code, header, table or
 * constant with the CUDA path.
 *
 * What it computes (paper: "LUNA: Linear Universal Neural Attention", arXiv
 * 2512.08061):
 *   - the feature map of Eq. (phi-def-scalarenv) with the default "no gate"
 *     envelope h = 1 of Sec. 5.4 / Table 5, scale 1/sqrt(M), projection bias b
 *     and per-channel scalar MLPs psi_l(u) = relu(fc2(relu(fc1(u)))) as in the
 *     appendix listing (TaskSpecificProjections, ScalarMLP, MLPLearnable-
 *     FeatureMap).  Feature index i*L + l (projection-major).
 *   - kernelized linear attention, Eq. (kernel-attn):
 *       O_i = phi(q_i)^T S / (phi(q_i)^T z + eps),  S = sum_j phi(k_j) v_j^T,
 *       z = sum_j phi(k_j); rows/keys at or beyond a sequence's valid length
 *       are excluded (keys) and produce 0 (queries).
 *   - the streaming (causal) form named in the abstract and Sec. 3.2: the same
 *     with the sums over j <= i, evaluated as a sequential prefix recurrence.
 *   - the brute-force quadratic form sum_j k(q_i,k_j) v_j / (sum_j k + eps)
 *     with k(x,y) = phi(x)^T phi(y) (Eq. kernel-attn read right to left).
 *   - the backward pass by the direct chain rule, sample by sample through
 *     every hidden unit of every channel MLP (ReLU'(0) taken as 0).
 *   - the listing's shared_channels variant: one scalar MLP with L outputs
 *     (fc1: 1 -> hid shared by the channels, fc2: hid -> L), so channel l
 *     reads the same hidden units with its own fc2 row.
 *   - the listing's nonneg = False: the channel outputs without the outer
 *     ReLU (features of either sign).
 *   - per-head parameters (the conversion experiments instantiate the feature
 *     map's parameters per layer and head, Sec. 5 / appendix): head h of every
 *     sequence uses its own W, b and channel MLPs; their gradients are summed
 *     over the batch only.
 *   - the feature-map variants of the kernel ablation (Sec. 5.4, Table 5) and
 *     the listing's ScalarMLP activation: a hidden-unit activation other
 *     than ReLU (GELU in its erf form, SiLU, tanh) evaluated directly; the
 *     envelope-gated map, channel l of every projection multiplied by the
 *     tokenwise gate h_l(x) = sigmoid(We_l . x + be_l) in [0, 1]; and
 *     Bank+Coef, channel l multiplied by a learned global coefficient c_l.
 *   - the listing's ch_rms channel normalisation: per call of the feature map
 *     (once over Q, once over K), every channel's MLP outputs are scaled by
 *     s_l = min(target / (rms_l + 1e-6), 1), rms_l = sqrt(mean y_l^2 + 1e-6)
 *     over every valid row and projection of that call's input; the backward
 *     pass carries the dependence of s_l on every output of the channel.
 *
 * Parity pinned by the CPU tests: hand-computed feature maps, the brute-force
 * quadratic form, closed-form special cases (constant channels give a plain
 * mean), the positive semi-definite Gram matrix of Prop. 1, invariances, and
 * central finite differences of the backward pass.
 */
#include <math.h>
#include <stddef.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>
#ifdef _OPENMP
#include <omp.h>
#endif

typedef struct {
    int d;            /* width of a query/key row                        */
    int M;            /* number of projections (rows of W)               */
    int L;            /* number of channel functions psi_l               */
    int hid;          /* hidden width of each channel MLP                */
    const double *W;  /* M x d                                           */
    const double *b;  /* M                                               */
    const double *w1; /* L x hid, fc1 weight of channel l (fan-in 1); hid if shared */
    const double *b1; /* L x hid; hid if shared                          */
    const double *w2; /* L x hid, fc2 weight of channel l (fan-out 1)    */
    const double *b2; /* L                                               */
    int shared;       /* 1: one MLP for all channels (fc1 shared)        */
    double ch_rms_target; /* > 0: channel RMS normalisation to this target */
    const double *chs;    /* per-channel scales s_l in effect (NULL: 1); set per input by the callers */
    int heads;            /* > 0: parameters per head (arrays carry a leading head axis of this size) */
    int signed_out;       /* 1: the listing's nonneg = False (no outer ReLU); 0: its default */
    int act;              /* hidden-unit activation: 0 ReLU (the default), 1 GELU (erf form), 2 SiLU, 3 tanh */
    const double *We;     /* L x d envelope gate weights (NULL: no gate, h = 1) */
    const double *be;     /* L envelope gate biases */
    const double *coef;   /* L Bank+Coef channel coefficients (NULL: 1) */
} oracle_phi;

/* Layout of oracle_phi, checked by the Python binding against its mirror of the struct. */
size_t oracle_phi_size(void) { return sizeof(oracle_phi); }
size_t oracle_phi_offset(int field) {
    switch (field) {
        case 0: return offsetof(oracle_phi, W);
        case 1: return offsetof(oracle_phi, shared);
        case 2: return offsetof(oracle_phi, ch_rms_target);
        case 3: return offsetof(oracle_phi, chs);
        case 4: return offsetof(oracle_phi, heads);
        case 5: return offsetof(oracle_phi, signed_out);
        case 6: return offsetof(oracle_phi, act);
        case 7: return offsetof(oracle_phi, We);
        case 8: return offsetof(oracle_phi, coef);
    }
    return (size_t)-1;
}

/* The parameters of head h: p itself, or with per-head parameters the h-th slice of every array. */
static oracle_phi head_view(const oracle_phi *p, int h) {
    oracle_phi q = *p;
    if (p->heads > 0) {
        const size_t n1 = (size_t)(p->shared ? 1 : p->L) * p->hid, n2 = (size_t)p->L * p->hid;
        q.W = p->W + (size_t)h * p->M * p->d;
        q.b = p->b + (size_t)h * p->M;
        q.w1 = p->w1 + (size_t)h * n1;
        q.b1 = p->b1 + (size_t)h * n1;
        q.w2 = p->w2 + (size_t)h * n2;
        q.b2 = p->b2 + (size_t)h * p->L;
        q.heads = 0;
    }
    return q;
}

/* offset of channel l's fc1 row (the one shared row when shared) */
static size_t fc1_row(const oracle_phi *p, int l) { return (size_t)(p->shared ? 0 : l) * p->hid; }

typedef struct {
    double *dW, *db, *dw1, *db1, *dw2, *db2;
    double *dWe, *dbe, *dcoef;  /* envelope and Bank+Coef parameters (NULL when the map has none) */
} oracle_grads;

static double relu(double x) { return x > 0.0 ? x : 0.0; }

/* The hidden-unit activation of the channel MLPs and its derivative (ReLU'(0) = 0).
 * GELU(a) = a Phi(a) with Phi the standard normal distribution function,
 * SiLU(a) = a sigma(a), tanh. */
#define ORACLE_PI 3.14159265358979323846
static double act_f(int act, double a) {
    switch (act) {
        case 1: return 0.5 * a * (1.0 + erf(a / sqrt(2.0)));
        case 2: return a / (1.0 + exp(-a));
        case 3: return tanh(a);
        default: return relu(a);
    }
}
static double act_df(int act, double a) {
    switch (act) {
        case 1: return 0.5 * (1.0 + erf(a / sqrt(2.0))) + a * exp(-0.5 * a * a) / sqrt(2.0 * ORACLE_PI);
        case 2: { const double sg = 1.0 / (1.0 + exp(-a)); return sg * (1.0 + a * (1.0 - sg)); }
        case 3: { const double t = tanh(a); return 1.0 - t * t; }
        default: return a > 0.0 ? 1.0 : 0.0;
    }
}

int oracle_max_threads(void) {
#ifdef _OPENMP
    return omp_get_max_threads();
#else
    return 1;
#endif
}

void oracle_set_threads(int t) {
#ifdef _OPENMP
    if (t > 0) omp_set_num_threads(t);
#else
    (void)t;
#endif
}

/* u_i = w_i^T x + b_i  (listing: TaskSpecificProjections.forward) */
static double project(const oracle_phi *p, int i, const double *x) {
    double u = p->b[i];
    for (int c = 0; c < p->d; ++c) u += p->W[(size_t)i * p->d + c] * x[c];
    return u;
}

/* y_l(u) = fc2(act(fc1(u))) before the non-negativity ReLU (listing: ScalarMLP) */
static double channel_pre(const oracle_phi *p, int l, double u) {
    const double *w1 = p->w1 + fc1_row(p, l);
    const double *b1 = p->b1 + fc1_row(p, l);
    const double *w2 = p->w2 + (size_t)l * p->hid;
    double y = p->b2[l];
    for (int k = 0; k < p->hid; ++k) y += w2[k] * act_f(p->act, w1[k] * u + b1[k]);
    return y;
}

/* psi_l(u): the channel output, through the outer ReLU unless the outputs are signed */
static double channel_out(const oracle_phi *p, int l, double u) {
    const double y = channel_pre(p, l, u);
    return p->signed_out ? y : relu(y);
}

double oracle_psi(const oracle_phi *p, int l, double u) { return channel_out(p, l, u); }

/* The envelope gate of channel l for the row x: h_l(x) = sigmoid(We_l . x + be_l), 1 without a gate. */
static double gate(const oracle_phi *p, int l, const double *x) {
    if (!p->We) return 1.0;
    double a = p->be[l];
    for (int c = 0; c < p->d; ++c) a += p->We[(size_t)l * p->d + c] * x[c];
    return 1.0 / (1.0 + exp(-a));
}

/* The Bank+Coef coefficient of channel l, 1 without one. */
static double chcoef(const oracle_phi *p, int l) { return p->coef ? p->coef[l] : 1.0; }

/* phi(x) = (1/sqrt(M)) [s_l h_l(x) c_l psi_l(w_i^T x + b_i)]_{i,l},  index i*L + l (s_l = 1 without
 * ch_rms, h_l = 1 without the envelope gate, c_l = 1 without Bank+Coef) */
static void phi_row(const oracle_phi *p, const double *x, double *out) {
    const double s = 1.0 / sqrt((double)p->M);
    for (int i = 0; i < p->M; ++i) {
        double u = project(p, i, x);
        for (int l = 0; l < p->L; ++l)
            out[i * p->L + l] = s * (p->chs ? p->chs[l] : 1.0) * gate(p, l, x) * chcoef(p, l) * channel_out(p, l, u);
    }
}

static int head_len(const int32_t *lengths, int b, int n);

/* Channel RMS statistics of one input X (B x H x n rows of width d; rows at or
 * past a sequence's length excluded): rms_l = sqrt(mean y_l^2 + 1e-6) over
 * every valid row and projection of the MLP outputs y_l = psi_l(u), the scale
 * s_l = min(target / (rms_l + 1e-6), 1), and the sample count N = rows x M.
 * The sums are taken head by head and added in head order. */
#define CH_RMS_EPS 1e-6
static void ch_rms_scales(const oracle_phi *p, const double *X, int B, int H, int n, const int32_t *lengths,
                          double *s, double *rms, double *count) {
    const int L = p->L, d = p->d, BH = B * H;
    double *part = (double *)calloc((size_t)(BH > 0 ? BH : 1) * L, sizeof(double));
    double rows = 0.0;
#pragma omp parallel for schedule(dynamic, 1)
    for (int bh = 0; bh < BH; ++bh) {
        const int len = head_len(lengths, bh / H, n);
        for (int r = 0; r < len; ++r) {
            const double *x = X + ((size_t)bh * n + r) * d;
            for (int i = 0; i < p->M; ++i) {
                const double u = project(p, i, x);
                for (int l = 0; l < L; ++l) {
                    const double y = channel_out(p, l, u);
                    part[(size_t)bh * L + l] += y * y;
                }
            }
        }
    }
    for (int bh = 0; bh < BH; ++bh) rows += head_len(lengths, bh / H, n);
    *count = rows * p->M;
    for (int l = 0; l < L; ++l) {
        double sum = 0.0;
        for (int bh = 0; bh < BH; ++bh) sum += part[(size_t)bh * L + l];
        const double mean = *count > 0.0 ? sum / *count : 0.0;
        rms[l] = sqrt(mean + CH_RMS_EPS);
        const double r = p->ch_rms_target / (rms[l] + CH_RMS_EPS);
        s[l] = r < 1.0 ? r : 1.0;
    }
    free(part);
}

void oracle_featmap(const oracle_phi *p0, const double *X, int64_t rows, double *Phi) {
    const int D = p0->M * p0->L;
    oracle_phi pc = *p0;
    const oracle_phi *p = &pc;
    double *sc = (double *)malloc(sizeof(double) * 3 * (size_t)p0->L);
    pc.chs = NULL;
    if (p0->ch_rms_target > 0.0) {  /* the statistics of this call's rows (all valid) */
        double cnt;
        ch_rms_scales(p0, X, 1, 1, (int)rows, NULL, sc, sc + p0->L, &cnt);
        pc.chs = sc;
    }
#pragma omp parallel for schedule(static)
    for (int64_t r = 0; r < rows; ++r) phi_row(p, X + r * p->d, Phi + r * D);
    free(sc);
}

/* Smallest relative distance of any ReLU argument of the feature map of a row
 * from its kink (inner hidden units and outer non-negativity ReLU).  Where it
 * is at rounding level the gradient of that row is not unique. */
void oracle_kink_margin(const oracle_phi *p, const double *X, int64_t rows, double *margin) {
#pragma omp parallel for schedule(static)
    for (int64_t r = 0; r < rows; ++r) {
        const double *x = X + r * p->d;
        double m = INFINITY;
        for (int i = 0; i < p->M; ++i) {
            double u = project(p, i, x);
            for (int l = 0; l < p->L; ++l) {
                const double *w1 = p->w1 + fc1_row(p, l);
                const double *b1 = p->b1 + fc1_row(p, l);
                const double *w2 = p->w2 + (size_t)l * p->hid;
                double y = p->b2[l], ysc = fabs(p->b2[l]);
                for (int k = 0; k < p->hid; ++k) {
                    double a = w1[k] * u + b1[k];
                    double sc = fabs(w1[k] * u) + fabs(b1[k]);
                    if (p->act == 0 && w1[k] != 0.0 && sc > 0.0) {  /* smooth activations have no kink */
                        double rel = fabs(a) / sc;
                        if (rel < m) m = rel;
                    }
                    y += w2[k] * act_f(p->act, a);
                    ysc += fabs(w2[k] * act_f(p->act, a));
                }
                if (ysc > 0.0 && !p->signed_out) {  /* the outer ReLU's kink */
                    double rel = fabs(y) / ysc;
                    if (rel < m) m = rel;
                }
            }
        }
        margin[r] = m;
    }
}

/* Backward of phi for `rows` rows: given dPhi, writes dX and accumulates the
 * parameter gradients into g, by the chain rule through every hidden unit. */
/* When set, the parameter gradients accumulate the absolute value of every
 * per-sample contribution instead (sum |term| of each gradient sum: the scale
 * of the rounding error of any finite-precision evaluation of that sum). */
static int abs_terms = 0;
void oracle_set_abs_terms(int on) { abs_terms = on ? 1 : 0; }
static double term(double v) { return abs_terms ? fabs(v) : v; }

/* With channel RMS normalisation (p->chs set), the gradient reaching the MLP
 * output y_l = psi_l(u) of one sample is (1/sqrt(M)) s_l dPhi + kappa_l y_l:
 * the first term through the scaled output, the second through s_l, which
 * depends on every sample of the channel (kappa from ch_rms_kappa). */
static void phi_rows_backward(const oracle_phi *p, const double *X, int64_t rows, const double *dPhi,
                              const double *kappa, double *dX, oracle_grads *g) {
    const int D = p->M * p->L, d = p->d, L = p->L;
    const double s = 1.0 / sqrt((double)p->M);
    double *h = (double *)malloc(sizeof(double) * 2 * (size_t)L);
    double *dE = h + L;  /* gradient with respect to e_l = h_l c_l of the row */
    for (int64_t r = 0; r < rows; ++r) {
        const double *x = X + r * d;
        double *dx = dX + r * d;
        for (int c = 0; c < d; ++c) dx[c] = 0.0;
        for (int l = 0; l < L; ++l) { h[l] = gate(p, l, x); dE[l] = 0.0; }
        for (int i = 0; i < p->M; ++i) {
            double u = project(p, i, x);
            double du = 0.0;
            for (int l = 0; l < L; ++l) {
                double y = channel_pre(p, l, u);
                const double dphi = dPhi[r * D + i * L + l];
                const double cs = p->chs ? p->chs[l] : 1.0;
                dE[l] += dphi * s * cs * (p->signed_out ? y : relu(y));
                if (!p->signed_out && !(y > 0.0)) continue; /* outer ReLU inactive */
                double dy = dphi * s * h[l] * chcoef(p, l);
                if (p->chs) dy = dy * p->chs[l] + (kappa ? kappa[l] * y : 0.0);
                if (dy == 0.0) continue;
                const double *w1 = p->w1 + fc1_row(p, l);
                const double *b1 = p->b1 + fc1_row(p, l);
                const double *w2 = p->w2 + (size_t)l * p->hid;
                g->db2[l] += term(dy);
                for (int k = 0; k < p->hid; ++k) {
                    double a = w1[k] * u + b1[k];
                    if (p->act == 0 && !(a > 0.0)) continue;  /* inactive ReLU unit */
                    g->dw2[(size_t)l * p->hid + k] += term(dy * act_f(p->act, a));
                    double dh = dy * w2[k] * act_df(p->act, a);
                    g->dw1[fc1_row(p, l) + k] += term(dh * u);  /* shared: summed over the channels */
                    g->db1[fc1_row(p, l) + k] += term(dh);
                    du += dh * w1[k];
                }
            }
            g->db[i] += term(du);
            for (int c = 0; c < d; ++c) {
                g->dW[(size_t)i * d + c] += term(du * x[c]);
                dx[c] += du * p->W[(size_t)i * d + c];
            }
        }
        /* e_l = h_l c_l: dc_l = dE_l h_l; through the gate, dh_l = dE_l c_l and
         * d(We_l . x + be_l) = dh_l h_l (1 - h_l) */
        for (int l = 0; l < L; ++l) {
            if (p->coef) g->dcoef[l] += term(dE[l] * h[l]);
            if (!p->We) continue;
            const double dpre = dE[l] * chcoef(p, l) * h[l] * (1.0 - h[l]);
            g->dbe[l] += term(dpre);
            for (int c = 0; c < d; ++c) {
                g->dWe[(size_t)l * d + c] += term(dpre * x[c]);
                dx[c] += dpre * p->We[(size_t)l * d + c];
            }
        }
    }
    free(h);
}

static int head_len(const int32_t *lengths, int b, int n) {
    if (!lengths) return n;
    int len = lengths[b];
    if (len < 0) len = 0;
    if (len > n) len = n;
    return len;
}

/* ------------------------------------------------------------------------ */
/* forward, linear (sufficient-statistics) form                              */

static void attn_fwd_head(const oracle_phi *pq_, const oracle_phi *pk_, int n, int dv, int causal, double eps,
                          const double *Q, const double *K, const double *V, int len, double *O) {
    const int D = pq_->M * pq_->L, d = pq_->d;
    double *phq = (double *)malloc(sizeof(double) * D);
    double *phk = (double *)malloc(sizeof(double) * D);
    double *S = (double *)calloc((size_t)D * dv, sizeof(double));
    double *z = (double *)calloc((size_t)D, sizeof(double));
    memset(O, 0, sizeof(double) * (size_t)n * dv);
    if (!causal) {
        for (int j = 0; j < len; ++j) {
            phi_row(pk_, K + (size_t)j * d, phk);
            for (int f = 0; f < D; ++f) {
                z[f] += phk[f];
                for (int c = 0; c < dv; ++c) S[(size_t)f * dv + c] += phk[f] * V[(size_t)j * dv + c];
            }
        }
    }
    for (int i = 0; i < len; ++i) {
        if (causal) { /* S_i = S_{i-1} + phi(k_i) v_i^T, z_i likewise */
            phi_row(pk_, K + (size_t)i * d, phk);
            for (int f = 0; f < D; ++f) {
                z[f] += phk[f];
                for (int c = 0; c < dv; ++c) S[(size_t)f * dv + c] += phk[f] * V[(size_t)i * dv + c];
            }
        }
        phi_row(pq_, Q + (size_t)i * d, phq);
        double den = eps;
        for (int f = 0; f < D; ++f) den += phq[f] * z[f];
        if (den == 0.0) continue;
        for (int c = 0; c < dv; ++c) {
            double num = 0.0;
            for (int f = 0; f < D; ++f) num += phq[f] * S[(size_t)f * dv + c];
            O[(size_t)i * dv + c] = num / den;
        }
    }
    free(phq); free(phk); free(S); free(z);
}

/* The feature maps applied to the queries and to the keys: both p itself, or,
 * with channel RMS normalisation, p with the scales of the statistics of all
 * valid query rows (pq) and of all valid key rows (pk).  st holds, per side,
 * s (L), rms (L) and the sample count N. */
typedef struct {
    oracle_phi pq, pk;
    double *st;
} side_maps;

static void side_maps_init(side_maps *sm, const oracle_phi *p, const double *Q, const double *K, int B, int H,
                           int n, const int32_t *lengths) {
    const int L = p->L;
    sm->pq = *p;
    sm->pk = *p;
    sm->pq.chs = sm->pk.chs = NULL;
    sm->st = (double *)calloc(2 * (2 * (size_t)L + 1), sizeof(double));
    if (p->ch_rms_target > 0.0) {
        double *sq = sm->st, *sk = sm->st + 2 * L + 1;
        ch_rms_scales(p, Q, B, H, n, lengths, sq, sq + L, sq + 2 * L);
        ch_rms_scales(p, K, B, H, n, lengths, sk, sk + L, sk + 2 * L);
        sm->pq.chs = sq;
        sm->pk.chs = sk;
    }
}

void oracle_attn_fwd(const oracle_phi *p, int B, int H, int n, int dv, int causal, double eps, const double *Q,
                     const double *K, const double *V, const int32_t *lengths, double *O) {
    const int d = p->d;
    side_maps sm;
    side_maps_init(&sm, p, Q, K, B, H, n, lengths);
#pragma omp parallel for schedule(dynamic, 1)
    for (int bh = 0; bh < B * H; ++bh) {
        int b = bh / H;
        size_t qo = (size_t)bh * n * d, vo = (size_t)bh * n * dv;
        const oracle_phi vq = head_view(&sm.pq, bh % H), vk = head_view(&sm.pk, bh % H);
        attn_fwd_head(&vq, &vk, n, dv, causal, eps, Q + qo, K + qo, V + vo, head_len(lengths, b, n), O + vo);
    }
    free(sm.st);
}

/* Channel RMS scales of the rows of X (B x H x n x d, valid rows only): s and rms (L each). */
void oracle_ch_rms(const oracle_phi *p, const double *X, int B, int H, int n, const int32_t *lengths, double *s,
                   double *rms) {
    double cnt;
    ch_rms_scales(p, X, B, H, n, lengths, s, rms, &cnt);
}

/* ------------------------------------------------------------------------ */
/* forward, brute-force quadratic form                                        */

void oracle_attn_quadratic(const oracle_phi *p, int B, int H, int n, int dv, int causal, double eps,
                           const double *Q, const double *K, const double *V, const int32_t *lengths,
                           double *O) {
    const int D = p->M * p->L, d = p->d;
    side_maps sm;
    side_maps_init(&sm, p, Q, K, B, H, n, lengths);
#pragma omp parallel for schedule(dynamic, 1)
    for (int bh = 0; bh < B * H; ++bh) {
        int len = head_len(lengths, bh / H, n);
        const double *q = Q + (size_t)bh * n * d, *k = K + (size_t)bh * n * d, *v = V + (size_t)bh * n * dv;
        double *o = O + (size_t)bh * n * dv;
        double *PQ = (double *)malloc(sizeof(double) * (size_t)(len > 0 ? len : 1) * D);
        double *PK = (double *)malloc(sizeof(double) * (size_t)(len > 0 ? len : 1) * D);
        const oracle_phi vq = head_view(&sm.pq, bh % H), vk = head_view(&sm.pk, bh % H);
        for (int i = 0; i < len; ++i) {
            phi_row(&vq, q + (size_t)i * d, PQ + (size_t)i * D);
            phi_row(&vk, k + (size_t)i * d, PK + (size_t)i * D);
        }
        memset(o, 0, sizeof(double) * (size_t)n * dv);
        for (int i = 0; i < len; ++i) {
            double den = eps;
            int jmax = causal ? i + 1 : len;
            double *acc = o + (size_t)i * dv;
            for (int j = 0; j < jmax; ++j) {
                double kij = 0.0; /* k(q_i, k_j) = phi(q_i)^T phi(k_j) */
                for (int f = 0; f < D; ++f) kij += PQ[(size_t)i * D + f] * PK[(size_t)j * D + f];
                den += kij;
                for (int c = 0; c < dv; ++c) acc[c] += kij * v[(size_t)j * dv + c];
            }
            if (den == 0.0) {
                for (int c = 0; c < dv; ++c) acc[c] = 0.0;
            } else {
                for (int c = 0; c < dv; ++c) acc[c] /= den;
            }
        }
        free(PQ); free(PK);
    }
    free(sm.st);
}

/* ------------------------------------------------------------------------ */
/* attention weights of a block of query rows (conversion, stage 1)          */

/* The attention distribution that the kernel induces, Eq. (kernel-attn) read
 * as a weighted average of the values: for query rows i in [row0, row0+rows)
 * of every (b, h),
 *     a_ij = k(q_i, k_j) / (sum_j' k(q_i, k_j') + eps),   k(x, y) = phi(x)^T phi(y),
 * over the valid keys j (j <= i in the streaming form), 0 for the other keys, for
 * query rows at or past the valid length, and for a row whose guarded sum is
 * exactly 0.  So O_i = sum_j a_ij v_j.  A is (B, H, rows, n).
 * With `teacher` non-zero, the softmax attention that the conversion distils
 * from instead (appendix, stage 1: the teacher is the original softmax module):
 *     p_ij = exp(q_i . k_j / sqrt(d)) / sum_j' exp(q_i . k_j' / sqrt(d))
 * over the same keys, with the same zero rows and columns. */
void oracle_attn_weights(const oracle_phi *p, int B, int H, int n, int causal, double eps, const double *Q,
                         const double *K, const int32_t *lengths, int row0, int rows, int teacher, double *A) {
    const int D = p->M * p->L, d = p->d;
    side_maps sm;
    side_maps_init(&sm, p, Q, K, B, H, n, lengths);
#pragma omp parallel for schedule(dynamic, 1)
    for (int bh = 0; bh < B * H; ++bh) {
        const int len = head_len(lengths, bh / H, n);
        const double *q = Q + (size_t)bh * n * d, *k = K + (size_t)bh * n * d;
        double *a = A + (size_t)bh * rows * n;
        memset(a, 0, sizeof(double) * (size_t)rows * n);
        double *pq = (double *)malloc(sizeof(double) * D);
        double *PK = (double *)malloc(sizeof(double) * (size_t)(len > 0 ? len : 1) * D);
        const oracle_phi vq = head_view(&sm.pq, bh % H), vk = head_view(&sm.pk, bh % H);
        for (int j = 0; j < len; ++j) phi_row(&vk, k + (size_t)j * d, PK + (size_t)j * D);
        for (int r = 0; r < rows; ++r) {
            const int i = row0 + r;
            if (i < 0 || i >= len) continue;
            const int jmax = causal ? i + 1 : len;
            double *ar = a + (size_t)r * n;
            if (teacher) {
                double mx = -INFINITY;
                for (int j = 0; j < jmax; ++j) {
                    double s = 0.0;
                    for (int c = 0; c < d; ++c) s += q[(size_t)i * d + c] * k[(size_t)j * d + c];
                    ar[j] = s / sqrt((double)d);
                    if (ar[j] > mx) mx = ar[j];
                }
                double tot = 0.0;
                for (int j = 0; j < jmax; ++j) {
                    ar[j] = exp(ar[j] - mx);
                    tot += ar[j];
                }
                for (int j = 0; j < jmax; ++j) ar[j] /= tot;
                continue;
            }
            phi_row(&vq, q + (size_t)i * d, pq);
            double den = eps;
            for (int j = 0; j < jmax; ++j) {
                double kij = 0.0;
                for (int f = 0; f < D; ++f) kij += pq[f] * PK[(size_t)j * D + f];
                ar[j] = kij;
                den += kij;
            }
            for (int j = 0; j < jmax; ++j) ar[j] = den == 0.0 ? 0.0 : ar[j] / den;
        }
        free(pq); free(PK);
    }
    free(sm.st);
}

/* ------------------------------------------------------------------------ */
/* backward                                                                  */

static void attn_bwd_head(const oracle_phi *pq_, const oracle_phi *pk_, int n, int dv, int causal, double eps,
                          const double *Q, const double *K, const double *V, const double *dO, int len, double *dQ,
                          double *dK, double *dV, oracle_grads *g, double *dPQ_out, double *dPK_out) {
    const int D = pq_->M * pq_->L, d = pq_->d;
    size_t nl = (size_t)(len > 0 ? len : 1);
    double *PQ = (double *)malloc(sizeof(double) * nl * D);
    double *PK = (double *)malloc(sizeof(double) * nl * D);
    double *dPQ = (double *)calloc(nl * D, sizeof(double));
    double *dPK = (double *)calloc(nl * D, sizeof(double));
    double *dnum = (double *)calloc(nl * dv, sizeof(double));
    double *dden = (double *)calloc(nl, sizeof(double));
    double *S = (double *)calloc((size_t)D * dv, sizeof(double));
    double *z = (double *)calloc((size_t)D, sizeof(double));
    double *o = (double *)malloc(sizeof(double) * dv);
    memset(dQ, 0, sizeof(double) * (size_t)n * d);
    memset(dK, 0, sizeof(double) * (size_t)n * d);
    memset(dV, 0, sizeof(double) * (size_t)n * dv);
    for (int i = 0; i < len; ++i) {
        phi_row(pq_, Q + (size_t)i * d, PQ + (size_t)i * D);
        phi_row(pk_, K + (size_t)i * d, PK + (size_t)i * D);
    }
    if (!causal) {
        for (int j = 0; j < len; ++j)
            for (int f = 0; f < D; ++f) {
                z[f] += PK[(size_t)j * D + f];
                for (int c = 0; c < dv; ++c) S[(size_t)f * dv + c] += PK[(size_t)j * D + f] * V[(size_t)j * dv + c];
            }
    }
    /* query side: o_i, dnum_i = do_i/den_i, dden_i = -(do_i . o_i)/den_i,
     * dphi(q_i) = S_i dnum_i + z_i dden_i */
    for (int i = 0; i < len; ++i) {
        if (causal)
            for (int f = 0; f < D; ++f) {
                z[f] += PK[(size_t)i * D + f];
                for (int c = 0; c < dv; ++c) S[(size_t)f * dv + c] += PK[(size_t)i * D + f] * V[(size_t)i * dv + c];
            }
        const double *pq = PQ + (size_t)i * D;
        double den = eps;
        for (int f = 0; f < D; ++f) den += pq[f] * z[f];
        if (den == 0.0) continue;
        double dot = 0.0;
        for (int c = 0; c < dv; ++c) {
            double num = 0.0;
            for (int f = 0; f < D; ++f) num += pq[f] * S[(size_t)f * dv + c];
            o[c] = num / den;
            dot += dO[(size_t)i * dv + c] * o[c];
        }
        dden[i] = -dot / den;
        for (int c = 0; c < dv; ++c) dnum[(size_t)i * dv + c] = dO[(size_t)i * dv + c] / den;
        for (int f = 0; f < D; ++f) {
            double acc = z[f] * dden[i];
            for (int c = 0; c < dv; ++c) acc += S[(size_t)f * dv + c] * dnum[(size_t)i * dv + c];
            dPQ[(size_t)i * D + f] = acc;
        }
    }
    /* key side: G_j = sum_{i >= j (or all i)} phi(q_i) dnum_i^T, g_j likewise with dden;
     * dv_j = G_j^T phi(k_j), dphi(k_j) = G_j v_j + g_j */
    double *G = S, *gz = z; /* reuse storage */
    memset(G, 0, sizeof(double) * (size_t)D * dv);
    memset(gz, 0, sizeof(double) * (size_t)D);
    if (!causal) {
        for (int i = 0; i < len; ++i)
            for (int f = 0; f < D; ++f) {
                gz[f] += PQ[(size_t)i * D + f] * dden[i];
                for (int c = 0; c < dv; ++c) G[(size_t)f * dv + c] += PQ[(size_t)i * D + f] * dnum[(size_t)i * dv + c];
            }
    }
    for (int j = len - 1; j >= 0; --j) {
        if (causal)
            for (int f = 0; f < D; ++f) {
                gz[f] += PQ[(size_t)j * D + f] * dden[j];
                for (int c = 0; c < dv; ++c) G[(size_t)f * dv + c] += PQ[(size_t)j * D + f] * dnum[(size_t)j * dv + c];
            }
        const double *pk = PK + (size_t)j * D;
        for (int c = 0; c < dv; ++c) {
            double acc = 0.0;
            for (int f = 0; f < D; ++f) acc += G[(size_t)f * dv + c] * pk[f];
            dV[(size_t)j * dv + c] = acc;
        }
        for (int f = 0; f < D; ++f) {
            double acc = gz[f];
            for (int c = 0; c < dv; ++c) acc += G[(size_t)f * dv + c] * V[(size_t)j * dv + c];
            dPK[(size_t)j * D + f] = acc;
        }
    }
    if (dPQ_out) {  /* channel RMS normalisation: the caller finishes the chain rule */
        memcpy(dPQ_out, dPQ, sizeof(double) * (size_t)len * D);
        memcpy(dPK_out, dPK, sizeof(double) * (size_t)len * D);
    } else {
        phi_rows_backward(pq_, Q, len, dPQ, NULL, dQ, g);
        phi_rows_backward(pk_, K, len, dPK, NULL, dK, g);
    }
    free(PQ); free(PK); free(dPQ); free(dPK); free(dnum); free(dden); free(S); free(z); free(o);
}

/* The gradient slots of one head's partial: [dW | db | dw1 | db1 | dw2 | db2 | dWe | dbe | dcoef]. */
static oracle_grads grads_at(const oracle_phi *p, double *base) {
    const size_t nW = (size_t)p->M * p->d, nb = p->M, nh = (size_t)p->L * p->hid, x = nW + nb + 3 * nh + p->L;
    oracle_grads g = {base, base + nW, base + nW + nb, base + nW + nb + nh, base + nW + nb + 2 * nh,
                      base + nW + nb + 3 * nh, base + x, base + x + (size_t)p->L * p->d,
                      base + x + (size_t)p->L * p->d + p->L};
    return g;
}

static void attn_bwd_all(const oracle_phi *p, int B, int H, int n, int dv, int causal, double eps, const double *Q,
                         const double *K, const double *V, const double *dO, const int32_t *lengths, double *dQ,
                         double *dK, double *dV, double *dW, double *db, double *dw1, double *db1, double *dw2,
                         double *db2, double *dWe, double *dbe, double *dcoef) {
    const int d = p->d, M = p->M, L = p->L, hid = p->hid;
    const size_t nW = (size_t)M * d, nb = M, nh = (size_t)L * hid, nb2 = L;
    const size_t per = nW + nb + 3 * nh + nb2 + (size_t)L * d + 2 * (size_t)L;
    const int BH = B * H, D = M * L;
    double *part = (double *)calloc((size_t)(BH > 0 ? BH : 1) * per, sizeof(double));
    side_maps sm;
    side_maps_init(&sm, p, Q, K, B, H, n, lengths);
    const int norm = p->ch_rms_target > 0.0;
    /* with channel RMS normalisation: dPhi of every valid row of both sides, kept for the second phase */
    double *dPQ = NULL, *dPK = NULL;
    if (norm) {
        dPQ = (double *)calloc((size_t)(BH > 0 ? BH : 1) * n * D, sizeof(double));
        dPK = (double *)calloc((size_t)(BH > 0 ? BH : 1) * n * D, sizeof(double));
    }
#pragma omp parallel for schedule(dynamic, 1)
    for (int bh = 0; bh < BH; ++bh) {
        oracle_grads g = grads_at(p, part + (size_t)bh * per);
        size_t qo = (size_t)bh * n * d, vo = (size_t)bh * n * dv, po = (size_t)bh * n * D;
        const oracle_phi vq = head_view(&sm.pq, bh % H), vk = head_view(&sm.pk, bh % H);
        attn_bwd_head(&vq, &vk, n, dv, causal, eps, Q + qo, K + qo, V + vo, dO + vo,
                      head_len(lengths, bh / H, n), dQ + qo, dK + qo, dV + vo, &g, norm ? dPQ + po : NULL,
                      norm ? dPK + po : NULL);
    }
    if (norm) {
        /* kappa_l = ds_l/drms_l * drms_l/dy (without the factor y) * A_l per side, where
         * A_l = sum over valid rows t and projections i of (1/sqrt(M)) dPhi_{t,i,l} y_{t,i,l};
         * s_l = target/(rms_l + eps) has ds/drms = -target/(rms_l + eps)^2 where not clamped,
         * and drms_l/dy = y/(N rms_l). */
        const double c = 1.0 / sqrt((double)M);
        double *A = (double *)calloc((size_t)(BH > 0 ? BH : 1) * 2 * L, sizeof(double));
        double *kappa = (double *)calloc(2 * (size_t)L, sizeof(double));
#pragma omp parallel for schedule(dynamic, 1)
        for (int bh = 0; bh < BH; ++bh) {
            const int len = head_len(lengths, bh / H, n);
            for (int side = 0; side < 2; ++side) {
                const double *X = (side ? K : Q) + (size_t)bh * n * d;
                const double *dP = (side ? dPK : dPQ) + (size_t)bh * n * D;
                double *a = A + ((size_t)bh * 2 + side) * L;
                const oracle_phi v = head_view(p, bh % H);
                for (int r = 0; r < len; ++r)
                    for (int i = 0; i < M; ++i) {
                        const double u = project(&v, i, X + (size_t)r * d);
                        for (int l = 0; l < L; ++l)
                            a[l] += c * dP[(size_t)r * D + i * L + l] * channel_out(&v, l, u);
                    }
            }
        }
        for (int side = 0; side < 2; ++side) {
            const double *st = sm.st + side * (2 * (size_t)L + 1);
            const double N = st[2 * L];
            for (int l = 0; l < L; ++l) {
                double a = 0.0;
                for (int bh = 0; bh < BH; ++bh) a += A[((size_t)bh * 2 + side) * L + l];
                const double rms = st[L + l];
                const double r = p->ch_rms_target / (rms + CH_RMS_EPS);
                kappa[side * L + l] = (N > 0.0 && r <= 1.0)
                                     ? -p->ch_rms_target / ((rms + CH_RMS_EPS) * (rms + CH_RMS_EPS)) / (N * rms) * a
                                     : 0.0;
            }
        }
#pragma omp parallel for schedule(dynamic, 1)
        for (int bh = 0; bh < BH; ++bh) {
            oracle_grads g = grads_at(p, part + (size_t)bh * per);
            const int len = head_len(lengths, bh / H, n);
            size_t qo = (size_t)bh * n * d, po = (size_t)bh * n * D;
            const oracle_phi vq = head_view(&sm.pq, bh % H), vk = head_view(&sm.pk, bh % H);
            phi_rows_backward(&vq, Q + qo, len, dPQ + po, kappa, dQ + qo, &g);
            phi_rows_backward(&vk, K + qo, len, dPK + po, kappa + L, dK + qo, &g);
        }
        free(A); free(kappa); free(dPQ); free(dPK);
    }
    free(sm.st);
    /* ordered reduction over the heads (fc1 gradients: hid entries when the MLP is shared); with
     * per-head parameters, head h's gradients are the sum over the batch of its units b*H + h */
    double *outs[9] = {dW, db, dw1, db1, dw2, db2, dWe, dbe, dcoef};
    const size_t n1 = p->shared ? (size_t)hid : nh, x = nW + nb + 3 * nh + nb2;
    size_t sizes[9] = {nW, nb, n1, n1, nh, nb2, (size_t)L * d, (size_t)L, (size_t)L};
    size_t offs[9] = {0, nW, nW + nb, nW + nb + nh, nW + nb + 2 * nh, nW + nb + 3 * nh, x, x + (size_t)L * d,
                      x + (size_t)L * d + L};
    const int G = p->heads > 0 ? H : 1;
    for (int t = 0; t < 9; ++t) {
        if (!outs[t]) continue;
        for (int h = 0; h < G; ++h)
            for (size_t e = 0; e < sizes[t]; ++e) {
                double acc = 0.0;
                for (int bh = 0; bh < BH; ++bh)
                    if (G == 1 || bh % H == h) acc += part[(size_t)bh * per + offs[t] + e];
                outs[t][(size_t)h * sizes[t] + e] = acc;
            }
    }
    free(part);
}

void oracle_attn_bwd(const oracle_phi *p, int B, int H, int n, int dv, int causal, double eps, const double *Q,
                     const double *K, const double *V, const double *dO, const int32_t *lengths, double *dQ,
                     double *dK, double *dV, double *dW, double *db, double *dw1, double *db1, double *dw2,
                     double *db2) {
    attn_bwd_all(p, B, H, n, dv, causal, eps, Q, K, V, dO, lengths, dQ, dK, dV, dW, db, dw1, db1, dw2, db2, NULL,
                 NULL, NULL);
}

/* oracle_attn_bwd with the gradients of the envelope gate (dWe: L x d, dbe: L) and of the Bank+Coef
 * coefficients (dcoef: L); each may be NULL when the map has no such parameters. */
void oracle_attn_bwd_var(const oracle_phi *p, int B, int H, int n, int dv, int causal, double eps, const double *Q,
                         const double *K, const double *V, const double *dO, const int32_t *lengths, double *dQ,
                         double *dK, double *dV, double *dW, double *db, double *dw1, double *db1, double *dw2,
                         double *db2, double *dWe, double *dbe, double *dcoef) {
    attn_bwd_all(p, B, H, n, dv, causal, eps, Q, K, V, dO, lengths, dQ, dK, dV, dW, db, dw1, db1, dw2, db2, dWe,
                 dbe, dcoef);
}
