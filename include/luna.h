/*
 * luna.h — C ABI of the GB300 (sm_103a) LUNA attention library.
 *
 * LUNA (arXiv 2512.08061) is kernelized linear attention with a learned
 * feature map
 *
 *     phi(x) = (1/sqrt(M)) [ psi_l(w_i^T x + b_i) ]_{i<M, l<L}  in R^{D},  D = M*L
 *
 * (Eq. phi-def-scalarenv with the default envelope h = 1 of Sec. 5.4 /
 * Table 5; projection bias b and feature index i*L + l as in the appendix
 * listing), where each channel function is a scalar ReLU MLP
 *
 *     psi_l(u) = relu( sum_k w2[l,k] relu(w1[l,k] u + b1[l,k]) + b2[l] )
 *
 * (listing: ScalarMLP with hidden width `hidden`, act = ReLU, nonneg = True,
 * one MLP per channel).  Attention is Eq. (kernel-attn):
 *
 *     O_i = phi(q_i)^T S / (phi(q_i)^T z + eps),  S = sum_j phi(k_j) v_j^T,  z = sum_j phi(k_j)
 *
 * with the sums over all valid keys (non-causal) or over j <= i (the streaming
 * form named in the abstract and Sec. 3.2).  S and z are the key-side
 * sufficient statistics S_KV and S_K1 of Sec. 4.
 *
 * Conventions for every entry point:
 *   - All tensor pointers are DEVICE pointers owned by the caller.  The
 *     library never allocates device memory and keeps no state between calls
 *     except a per-process cache of the driver entry point it needs for TMA.
 *   - Q, K, dQ, dK are contiguous (B, H, n, d); V, O, dO, dV are contiguous
 *     (B, H, n, dv), element type `io` (fp32 or bf16).  Row-major, C order.
 *   - `lengths` is NULL (every sequence has n valid tokens) or a device array
 *     of B int32 valid lengths (right padding).  Values are clamped to [0, n].
 *     Keys at or beyond the length do not enter S and z; query rows at or
 *     beyond it produce O = 0 and receive dQ = dK = dV = 0.
 *   - `stream` is a cudaStream_t passed as void* (NULL = legacy default stream).
 *     Every call only enqueues work on it and returns without synchronising.
 *   - Argument errors are reported before anything is launched.  A failed
 *     launch returns LUNA_ERR_CUDA.  Device-side bounded waits that gave up
 *     are reported by luna_device_status().
 *   - Computation: the feature map is evaluated in fp32 for both io types
 *     (the listing casts the projections to float before the channel MLPs).
 *     Accumulations are fp32.  With io = bf16 the tensor-core contractions take
 *     bf16 operands; the normaliser phi(q)^T z is always an fp32 dot product.
 */
#ifndef LUNA_H
#define LUNA_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
    LUNA_OK = 0,
    LUNA_ERR_INVALID_ARG = 1,    /* NULL pointer, negative size, bad enum            */
    LUNA_ERR_UNSUPPORTED = 2,    /* valid but outside the supported shape range     */
    LUNA_ERR_WORKSPACE = 3,      /* workspace / table / state buffer too small      */
    LUNA_ERR_CUDA = 4,           /* a CUDA runtime call or launch failed            */
    LUNA_ERR_DEVICE_TIMEOUT = 5  /* a bounded device-side wait gave up              */
} luna_status;

typedef enum { LUNA_F32 = 0, LUNA_BF16 = 1 } luna_dtype;

/* Hidden-unit activation of the channel MLPs (the listing's ScalarMLP `act`):
 * ReLU is the listing's default and the only one with the exact
 * piecewise-linear table; the others are evaluated directly.
 * GELU(a) = a Phi(a) (Phi: the standard normal distribution function, the erf
 * form), SiLU(a) = a / (1 + e^-a), tanh. */
typedef enum { LUNA_ACT_RELU = 0, LUNA_ACT_GELU = 1, LUNA_ACT_SILU = 2, LUNA_ACT_TANH = 3 } luna_act;

/* Shape of the feature map (Eq. phi-def-scalarenv; listing defaults hidden = 64).
 * shared_channels = 0: one scalar MLP per channel (the listing's default);
 * 1: one scalar MLP with L outputs serves all channels (the listing's
 * shared_channels = True: fc1 Linear(1, hidden) shared, fc2 Linear(hidden, L)).
 * ch_rms_target > 0 turns on the listing's channel RMS normalisation
 * (ch_rms): each application of the feature map, once to all queries and once
 * to all keys of the batch, scales channel l of the MLP outputs y_l by
 * s_l = min(target / (rms_l + 1e-6), 1), rms_l = sqrt(mean y_l^2 + 1e-6) over
 * every valid row (rows at or past a sequence's length excluded) and every
 * projection; the backward pass includes the dependence of s_l on every
 * sample.  0 = off (the listing's default); negative, NaN or infinite is
 * LUNA_ERR_INVALID_ARG.  With it on, luna_attn_fwd / luna_attn_bwd support
 * both forms (the streaming form runs on a copy of the table, in the
 * workspace, whose channel-l coefficients are scaled by sqrt(s^q_l s^k_l));
 * luna_featmap, luna_attn_decode and luna_attn_weights give
 * LUNA_ERR_UNSUPPORTED (a batch statistic has no single-row or single-token
 * form).
 * signed_outputs = 1 is the listing's ScalarMLP(nonneg = False): the channel
 * outputs are fc2(relu(fc1(u))) without the outer ReLU, so features (and kernel
 * values) of either sign; 0 keeps the outer ReLU (the listing's default).  The
 * table is the same for both (the flag is read from the descriptor by every
 * call, so pass the same descriptor to all calls of one problem); with
 * ch_rms_target > 0 it gives LUNA_ERR_UNSUPPORTED.
 * param_head_stride = 0: one parameter set serves every head (the listing's
 * "shared ... over tokens/heads").  > 0: per-head parameters, as in the
 * conversion of a pretrained model, where the feature map's parameters are
 * instantiated per layer and head (appendix, conversion of BERT and ViT):
 * `table` holds ad->H tables, head h's at table + h * param_head_stride bytes
 * (each prepared by luna_phi_prepare from head h's parameters; the stride is
 * at least luna_phi_table_size and a multiple of 256), and luna_attn_bwd
 * writes each head's parameter gradients, summed over the batch only, as
 * arrays with a leading head axis (dW [H][M][d], ..., db2 [H][L]).  The
 * attention calls then run one sub-problem per head index (the B sequences'
 * head h at a time).  Not with ch_rms_target > 0 (LUNA_ERR_UNSUPPORTED); for
 * luna_featmap pass head h's table with a stride of 0.
 * Feature-map variants (the kernel ablation of Sec. 5.4, Table 5; each 0 = off,
 * the paper's default "no gate" map psi):
 *   act (a luna_act): the channel MLPs' hidden activation.  Not ReLU: every
 *     (row, projection) evaluates the L channel MLPs unit by unit, and the
 *     backward pass sums the MLP parameter gradients sample by sample (the
 *     interval histogram needs a piecewise-linear MLP).
 *   envelope = 1: the envelope-gated map phi(x) = h(x) (.) psi(x), channel l
 *     of every projection multiplied by the tokenwise gate
 *     h_l(x) = sigmoid(We_l . x + be_l) in (0, 1) (We, be in luna_phi_params;
 *     their gradients dWe, dbe in luna_phi_grads).
 *   bank_coef = 1: Bank+Coef, channel l of every projection multiplied by a
 *     learned global coefficient c_l (coef; gradient dcoef): an input-agnostic
 *     reweighting of the bank of channel functions that keeps the feature
 *     dimension M*L (a negative c_l gives features of either sign).
 *   They combine with each other and with shared_channels and signed_outputs;
 *   any of them runs the attention calls on the generic (CUDA-core) kernels and
 *   gives LUNA_ERR_UNSUPPORTED with ch_rms_target > 0, with param_head_stride,
 *   and in luna_attn_decode and luna_attn_weights.  The
 *   table holds the gate and coefficient parameters, so pass the same
 *   descriptor to every call of one problem.
 * Supported: 1 <= M, 1 <= L <= 16, M*L <= 128, 1 <= hidden <= 128, L*hidden <= 512. */
typedef struct {
    int M;               /* number of projections w_i (rows of W)       */
    int L;               /* number of channel functions psi_l           */
    int hidden;          /* hidden width of each (or the shared) MLP     */
    int shared_channels; /* 0 or 1, see above                           */
    float ch_rms_target; /* channel RMS normalisation target, 0 = off   */
    int signed_outputs;  /* 0 or 1, see above                           */
    int64_t param_head_stride; /* bytes between heads' tables, 0 = shared  */
    int act;             /* luna_act of the channel MLPs' hidden units   */
    int envelope;        /* 0 or 1: envelope-gated map, see above        */
    int bank_coef;       /* 0 or 1: Bank+Coef channel coefficients       */
} luna_phi_desc;

/* Feature-map parameters, fp32 device arrays, row-major:
 *   W [M][d], b [M], w1 [L][hidden], b1 [L][hidden], w2 [L][hidden], b2 [L];
 *   with shared_channels, w1 and b1 are [hidden] (the one fc1).
 * w1[l][k], b1[l][k] are fc1 of channel l (Linear(1, hidden)); w2[l][k], b2[l]
 * are its fc2 (Linear(hidden, 1)), or row l of the shared fc2. The same
 * parameters serve queries and keys and are shared by all heads (listing:
 * "shared ... over tokens/heads").  The variants' parameters: We [L][d], be [L]
 * (envelope gate; read only with envelope = 1) and coef [L] (read only with
 * bank_coef = 1); NULL when their variant is off. */
typedef struct {
    const float *W, *b, *w1, *b1, *w2, *b2;
    const float *We, *be, *coef;
} luna_phi_params;

/* Gradients of the feature-map parameters, fp32 device arrays with the shapes
 * of luna_phi_params (dw1, db1 of [hidden] with shared_channels).  They are
 * OVERWRITTEN (not accumulated) by luna_attn_bwd.  dWe, dbe (envelope = 1) and
 * dcoef (bank_coef = 1) are required with their variant and ignored without. */
typedef struct {
    float *dW, *db, *dw1, *db1, *dw2, *db2;
    float *dWe, *dbe, *dcoef;
} luna_phi_grads;

/* Problem description (Sec. 3.1: Q, K in R^{n x d}; Sec. 4: values of width d_v).
 * Supported: 1 <= d, dv <= 128; B, H, n >= 0 (an empty problem is a no-op).
 * causal = 1 selects the streaming form (sums over j <= i).  chunk (0, or
 * 16..128 in steps of 16, else LUNA_ERR_INVALID_ARG) is accepted for the
 * interface and otherwise not used: the kernels choose their own tiles (128
 * rows in the tensor-core streaming forward, 64 in its backward, 16 in the
 * generic kernels), and results do not depend on it beyond rounding order.
 * eps >= 0 guards the row normaliser: O_i = num_i / (den_i + eps); a row
 * whose guarded normaliser is exactly 0 produces O_i = 0 and zero gradients. */
typedef struct {
    int B, H, n, d, dv;
    int causal;
    int chunk;
    float eps;
    luna_dtype io;
} luna_attn_desc;

/* Human-readable name of a status code (static string, never NULL). */
const char *luna_status_string(luna_status s);

/* Bytes of the prepared feature-map table for this descriptor and input width d
 * (written to *bytes).  The table is an opaque device blob produced by
 * luna_phi_prepare and consumed by every other call. */
luna_status luna_phi_table_size(const luna_phi_desc *pd, int d, size_t *bytes);

/* Builds the feature-map table from the parameters (Eq. phi-def-scalarenv,
 * listing ScalarMLP): a copy of W and b, and for every channel the exact
 * piecewise-linear form of psi_l.  A ReLU MLP of a scalar is linear between
 * the kinks t = -b1/w1 of its hidden units, so on the merged, sorted kink list
 * psi_l(u) = relu(alpha_{l,j} u + beta_{l,j}) on interval j.  Kinks are
 * placed at the exact fp32 thresholds of fma(w1, u, b1) > 0, so the interval
 * decides every hidden unit exactly as an fp32 evaluation of fc1 would.
 * With a non-ReLU act the table still holds the parameters (the calls
 * evaluate the MLPs from them) and the piecewise form is not used; with
 * envelope or bank_coef it also holds We, be or coef.
 * `table` is a device buffer of at least luna_phi_table_size bytes, 256-byte
 * aligned; it must not be modified while a call that reads it is in flight.
 * Parameters must be finite. */
luna_status luna_phi_prepare(const luna_phi_desc *pd, int d, const luna_phi_params *params, void *table,
                             size_t table_bytes, void *stream);

/* phi(X) for `rows` rows of width d (Eq. phi-def-scalarenv).
 * X: device, rows x d of type `xtype`; Phi: device fp32, rows x (M*L), feature
 * index i*L + l.  Debug / interoperability entry point: the attention calls
 * never materialise phi in memory. */
luna_status luna_featmap(const luna_phi_desc *pd, int d, const void *table, const void *X, luna_dtype xtype,
                         int64_t rows, float *Phi, void *stream);

/* Bytes of scratch memory the calls need (written to *bytes).  `backward`
 * selects the requirement of luna_attn_bwd (0 = luna_attn_fwd).  The caller
 * owns the workspace; its contents on entry are irrelevant and on exit are
 * unspecified.  Must be 256-byte aligned. */
luna_status luna_workspace_size(const luna_attn_desc *ad, const luna_phi_desc *pd, int backward, size_t *bytes);

/* Bytes of the optional forward state (the key statistics S, z of Sec. 4 per
 * head; for the causal form, the prefix statistics at every state segment). */
luna_status luna_state_size(const luna_attn_desc *ad, const luna_phi_desc *pd, size_t *bytes);

/* Forward pass, Eq. (kernel-attn) (causal: streaming form).
 * Q, K, V, lengths, O as in the conventions above.  `table` from
 * luna_phi_prepare.  `state` is NULL or a device buffer of luna_state_size
 * bytes that receives the key statistics for a later luna_attn_bwd.
 * `workspace` holds ws_bytes >= luna_workspace_size(ad, pd, 0). */
luna_status luna_attn_fwd(const luna_attn_desc *ad, const luna_phi_desc *pd, const void *table, const void *Q,
                          const void *K, const void *V, const int32_t *lengths, void *O, void *state,
                          void *workspace, size_t ws_bytes, void *stream);

/* Backward pass of luna_attn_fwd: given dO = dLoss/dO, writes dQ, dK, dV and
 * the parameter gradients `grads` (overwritten) of the same loss.
 * `state` is NULL (the key statistics are recomputed from K and V) or the
 * state written by luna_attn_fwd on the same Q, K, V, lengths and table.
 * The derivative of each ReLU at 0 is taken as 0.  Parameter gradients are
 * summed over all heads, rows and projections.  With pd->ch_rms_target > 0 the
 * channel statistics of Q and K are recomputed by every call, and a `state`
 * must come from luna_attn_fwd with the same descriptors (it holds the
 * normalised key statistics). */
luna_status luna_attn_bwd(const luna_attn_desc *ad, const luna_phi_desc *pd, const void *table, const void *Q,
                          const void *K, const void *V, const void *dO, const int32_t *lengths,
                          const void *state, void *dQ, void *dK, void *dV, const luna_phi_grads *grads,
                          void *workspace, size_t ws_bytes, void *stream);

/* Attention weights of query rows [row0, row0 + rows) of every (b, h), for the
 * conversion of a softmax model (appendix, "Stage 1: attention distillation":
 * the feature-map parameters are trained so that the attention distribution the
 * kernel induces matches the one of the original softmax module; the paper
 * does not fix the loss, so this call only produces the distributions).
 *   teacher = 0: the LUNA weights, Eq. (kernel-attn) read as a weighted average
 *       of the values,  a_ij = k(q_i, k_j) / (sum_j' k(q_i, k_j') + eps),
 *       k(x, y) = phi(x)^T phi(y), so that O_i = sum_j a_ij v_j exactly;
 *   teacher = 1: the softmax weights of the same queries and keys,
 *       p_ij = exp(q_i . k_j / sqrt(d)) / sum_j' exp(q_i . k_j' / sqrt(d))
 *       (`table` may then be NULL).
 * The sums run over the valid keys (j <= i with ad->causal = 1).  Keys outside
 * them, query rows at or past the valid length, and rows whose guarded sum is
 * exactly 0 get weight 0.  Q, K as in the conventions (ad->dv and ad->chunk are
 * ignored); A: fp32 device array (B, H, rows, n), every entry written.
 * 0 <= row0, 0 <= rows, row0 + rows <= n, else LUNA_ERR_INVALID_ARG;
 * pd->ch_rms_target > 0 gives LUNA_ERR_UNSUPPORTED.  No workspace: each block
 * of 32 rows writes its raw scores and normalises them in a second pass over
 * its own rows.  The feature map is fp32 for both io types; each row's sum
 * is accumulated in fp64. */
luna_status luna_attn_weights(const luna_attn_desc *ad, const luna_phi_desc *pd, const void *table, const void *Q,
                              const void *K, const int32_t *lengths, int row0, int rows, int teacher, float *A,
                              void *stream);

/* Location of the final state of a streaming-form forward pass (ad->causal = 1)
 * inside a `state` buffer written by luna_attn_fwd: the key statistics over all
 * valid tokens of each sequence, S = sum_j phi(k_j) v_j^T and z = sum_j phi(k_j)
 * (Eq. kernel-attn, streaming form of Sec. 3.2).  Head (b, h) holds S at
 * *S + (b*H + h) * *S_stride (D x dv fp32, row-major) and z at
 * *z + (b*H + h) * *z_stride (D fp32).  No device memory is touched; the
 * pointers are for luna_attn_decode, which continues each sequence after its
 * last valid token.  LUNA_ERR_INVALID_ARG for a non-causal descriptor or NULL
 * arguments. */
luna_status luna_state_final(const luna_attn_desc *ad, const luna_phi_desc *pd, void *state, float **S,
                             int64_t *S_stride, float **z, int64_t *z_stride);

/* One step of the streaming form (recurrent decode; the abstract and Sec. 3.2
 * name the associative streaming form of Eq. kernel-attn): for every (b, h)
 * and the new token's q, k, v,
 *     S <- S + phi(k) v^T,   z <- z + phi(k),   o = phi(q)^T S / (phi(q)^T z + eps)
 * i.e. the causal output of the token that follows the state's tokens.
 * q, k: (B, H, d); v, o: (B, H, dv), element type ad->io, one token per
 * (b, h); ad->n, ad->causal and ad->chunk are ignored.  S, z: fp32 device
 * arrays updated in place, head (b, h) at S + (b*H + h) * S_stride ([D][dv]
 * row-major) and z + (b*H + h) * z_stride ([D]); a stride of 0 selects the
 * dense layout (D*dv, D), a smaller nonzero stride is LUNA_ERR_INVALID_ARG.
 * A head whose guarded normaliser is exactly 0 produces o = 0.  No workspace;
 * B*H = 0 is a no-op. */
luna_status luna_attn_decode(const luna_attn_desc *ad, const luna_phi_desc *pd, const void *table, const void *q,
                             const void *k, const void *v, void *o, float *S, int64_t S_stride, float *z,
                             int64_t z_stride, void *stream);

/* Synchronises `stream`, then reads and clears the device status word at the
 * start of `workspace`.  Every luna_attn_fwd / luna_attn_bwd call clears the
 * word when it starts; a device-side wait of that call that ran out of its
 * iteration limit sets it (the kernel then abandons its work and returns, so
 * the outputs of that call are undefined).  So this reports the LAST call that
 * used this workspace: LUNA_OK, LUNA_ERR_DEVICE_TIMEOUT, or LUNA_ERR_CUDA if
 * synchronising or the copy failed (including an earlier asynchronous fault). */
luna_status luna_device_status(void *workspace, void *stream);

/* Diagnostic of the failure path (not needed for computation): launches one
 * block that waits on a device-side barrier phase nothing ever completes,
 * gives up after limit_ns nanoseconds of wall time (1 <= limit_ns <= 1e9) and
 * sets the status word at the start of `workspace` exactly as a kernel of
 * luna_attn_fwd / luna_attn_bwd whose bounded wait ran out does.  A following
 * luna_device_status(workspace) then reports LUNA_ERR_DEVICE_TIMEOUT and clears
 * the word; the CUDA context stays usable and later calls run normally.
 * `workspace` as for luna_attn_fwd (256-byte aligned); LUNA_ERR_INVALID_ARG for
 * NULL or a limit out of range. */
luna_status luna_selftest_wait(void *workspace, int64_t limit_ns, void *stream);

/* Size of the library-owned scratch array used by luna_attn_fwd_noalloc. */
#define LUNA_NOALLOC_SCRATCH_BYTES (16u << 20)

/* luna_attn_fwd without a caller-provided workspace.  The paper has no
 * counterpart; this is a deployment convenience.
 *
 * Some callers hold only their input and output buffers and have no way to
 * obtain device scratch memory: a custom operator inside an inference engine
 * whose device-memory plan is fixed before it runs and that is handed nothing
 * but its tensors, or host code that must not call into an allocator while it
 * runs (fixed-latency loops).  For them this entry point allocates nothing:
 * no cudaMalloc, cudaFree or allocating library routine is called.  Its
 * scratch is one file-scope __device__ array of LUNA_NOALLOC_SCRATCH_BYTES
 * (16 MiB) that every GPU which loads the library holds until the process
 * exits; problems whose forward workspace (luna_workspace_size with
 * backward = 0) exceeds it are rejected with LUNA_ERR_WORKSPACE before
 * anything is launched.  Arguments and results are those of luna_attn_fwd
 * with state = NULL (no key statistics are kept for a backward pass).
 *
 * The first call on a device, with that device current, looks up the array's
 * device address (cudaGetSymbolAddress) and caches it; make that first call
 * before any stream capture.  All calls in the process share the one array
 * per device and leave their contents in it; each call clears what must start
 * at zero.  Calls whose executions overlap on the GPU (different streams, or
 * different host threads) race on the array and give undefined results: order
 * them on one stream.  The cached address is that of the device's primary
 * context: after cudaDeviceReset the array may move, and the library must not
 * be used on that device again in the same process.
 *
 * A bounded device-side wait of the call that ran out sets the status word at
 * the start of the array, as luna_attn_fwd does in its workspace (O is then
 * undefined); the next call clears it.  luna_noalloc_scratch gives the array's
 * address, so that luna_device_status(scratch, stream) reports the status of
 * the last call on the device. */
luna_status luna_attn_fwd_noalloc(const luna_attn_desc *ad, const luna_phi_desc *pd, const void *table,
                                  const void *Q, const void *K, const void *V, const int32_t *lengths, void *O,
                                  void *stream);

/* Device address and size of the scratch array of luna_attn_fwd_noalloc on the
 * current device (the same set-up as that call's first use: make the first call
 * before any stream capture).  Allocates nothing.  The address serves
 * luna_device_status, which reads and clears the status word of the last
 * luna_attn_fwd_noalloc call on this device, and luna_selftest_wait; the rest of
 * the array is the no-allocation call's scratch and must not be written while
 * such a call may be in flight.  The paper has no counterpart.
 * LUNA_ERR_INVALID_ARG for NULL arguments, LUNA_ERR_CUDA if the lookup fails. */
luna_status luna_noalloc_scratch(void **scratch, size_t *bytes);

/* Kernel timing (tracing aid, not needed for computation).  After
 * luna_profile_start(name), every launch of the library kernel `name` (e.g.
 * "bwd_query", "keystats"; the names are listed in the library's kernel
 * launch sites) is bracketed by two CUDA events recorded on the stream it is
 * launched on, up to 4096 launches.  luna_profile_stop waits for the recorded
 * events and returns the summed launch durations in milliseconds and the
 * number of launches, then stops recording.  Process-wide; one kernel name at
 * a time. */
luna_status luna_profile_start(const char *kernel);
luna_status luna_profile_stop(double *total_ms, int *launches);

/* Number of kernels this library has launched in this process since it was
 * loaded (all entry points, all streams). */
uint64_t luna_launch_count(void);

/* Library version, e.g. 100 for 0.1.0. */
int luna_version(void);

#ifdef __cplusplus
}
#endif

#endif /* LUNA_H */
