/*
 * bom.h - C ABI of the GB300-native BOM (Backpropagated Output Momentum)
 *         task-space momentum pass.
 *
 * One optimizer step of BOM (paper, Algorithm 1) splits into two calls:
 *
 *   bom_step    forward through the backbone and the linear head, the
 *               residuals r_i = softmax(z_i) - onehot(y_i), their batch mean
 *               s_t over the supervised set I_t, the task-space EMA
 *               q_t = beta1 q_{t-1} + (1-beta1) s_t with qhat_t = q_t/(1-beta1^t),
 *               and ONE backward pass of the logit cotangent
 *               N_t^-1 [(1-lambda) r_i + lambda qhat_t], which yields the
 *               update numerator u = (1-lambda) g + lambda Jbar^T qhat for
 *               every tensor (Section 3.2, Eq. mix-objective and Eq. mix-gradient;
 *               LM construction appendix for I_t and N_t).
 *   bom_update  v = beta2 v + (1-beta2) u^2, vhat = v/(1-beta2^t),
 *               theta <- (1 - lr*wd) theta - lr u/(sqrt(vhat)+eps)
 *               (Section 3.4; Algorithm 1, last two steps).  No first-moment
 *               state exists and no first-moment bias correction is applied.
 *
 * Conventions shared by every entry point
 * ---------------------------------------
 * - Every tensor argument is a caller-owned DEVICE pointer (cudaMalloc or a
 *   PyTorch CUDA tensor), row-major and dense, unless stated otherwise.  The
 *   library never frees or keeps caller pointers beyond the call.
 * - bf16 values are passed as raw 16-bit patterns (uint16_t / void*).
 * - `stream` is a cudaStream_t passed as void*; NULL means the legacy default
 *   stream.  All work is enqueued asynchronously on it; no entry point except
 *   bom_get_stats synchronises.
 * - Host-checkable problems (null pointers, bad sizes, t < 1, unaligned
 *   pointers) return an error immediately and enqueue nothing.  Problems only
 *   the device can see (a bad label, N_t = 0, non-finite logits, a device step
 *   counter below 1, a bounded wait that ran out) are latched in a device
 *   status word of the handle; every later kernel of the step skips its work,
 *   q (and, with the fused update, every parameter and v) is left unmodified,
 *   and bom_get_stats returns the latched code.  The word is cleared at the
 *   start of each bom_step.
 * - Kernels are launched with programmatic dependent launch: a kernel may be
 *   scheduled while the previous one on the stream finishes, but it waits for
 *   that one's completion before touching memory, so stream order holds for
 *   the caller's own work before and after every call.
 * - Alignment: every bf16 tensor used by the tensor-core path needs a 16-byte
 *   aligned base and a row length that is a multiple of 8 elements (TMA rule);
 *   otherwise BOM_ENOTSUP.
 */
#ifndef BOM_H
#define BOM_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
    BOM_OK = 0,
    BOM_EINVAL = 1,    /* bad argument (host-detected, nothing enqueued)             */
    BOM_ENOMEM = 2,    /* workspace allocation failed                                 */
    BOM_ECUDA = 3,     /* a CUDA runtime / driver call failed                         */
    BOM_ELABEL = 4,    /* device: a label outside [0, d_out) that is not ignore_index */
    BOM_EEMPTY = 5,    /* device: N_t = 0 (Algorithm 1 requires N_t > 0)              */
    BOM_ETIMEOUT = 6,  /* device: a bounded wait inside a kernel ran out              */
    BOM_ENOTSUP = 7,   /* shape or alignment this build does not handle               */
    BOM_ENONFINITE = 8, /* a row's log-sum-exp or its label logit is not finite
                           (device-detected before any state is written)             */
    BOM_ESHARD = 9      /* device: another shard of a sharded step latched an error
                           (bom_step_shard_end, bom_step_vshard_mid), so this
                           shard stopped too                                        */
} bom_status;

typedef enum { BOM_F32 = 0, BOM_BF16 = 1 } bom_dtype;

typedef enum {
    BOM_LAYER_LINEAR = 0,       /* y = x W^T (+ b)                                         */
    BOM_LAYER_LINEAR_GELU = 1,  /* y = GELU(x W^T (+ b)), exact erf GELU                  */
    BOM_LAYER_SWIGLU = 2,       /* y = x + W_d (SiLU(x W_g^T) * (x W_u^T)); d_out = ffn    */
    BOM_LAYER_RMSNORM = 3       /* y = x / sqrt(mean_j x_j^2 + 1e-6) * gamma; d_out = d_in,
                                   no bias (the norm tensors of the language-model setting) */
} bom_layer_kind;

typedef enum {
    BOM_OUT_U = 0,        /* one backward pass: grads[] receive u                        */
    BOM_OUT_G_AND_H = 1   /* diagnostic: grads[] receive g (cotangent r_i/N_t) and      */
                          /* h_out[] receive h = Jbar^T qhat (cotangent qhat/N_t)       */
} bom_out_mode;

typedef struct {
    int32_t kind;      /* bom_layer_kind                                                */
    int32_t has_bias;  /* LINEAR / LINEAR_GELU: 1 adds a bias of length d_out           */
    int64_t d_in;      /* input width                                                   */
    int64_t d_out;     /* output width (SWIGLU: the ffn width; output stays d_in)       */
} bom_layer;

typedef struct {
    int64_t max_rows;         /* largest n_rows bom_step accepts (sizes the workspace)   */
    int64_t d_in;             /* width of the input X                                   */
    int64_t d_out;            /* classes / vocabulary size (head output width)          */
    int32_t n_layers;         /* backbone layers before the head (0 = head only)        */
    const bom_layer* layers;  /* host array of n_layers entries, copied by bom_init     */
    int32_t head_bias;        /* 1: the head has a bias of length d_out                 */
    int32_t compute;          /* bom_dtype of X, parameters and grads                   */
    float lambda;             /* mixture weight (paper default 0.5)                     */
    float beta1;              /* task-space EMA decay (paper default 0.9)               */
    int32_t ignore_index;     /* label value excluded from I_t (usually -100)           */
    int32_t out_mode;         /* bom_out_mode                                           */
} bom_config;

typedef struct {
    float loss;          /* mean cross-entropy over I_t                               */
    int32_t n_t;         /* |I_t|                                                     */
    int32_t status;      /* bom_status latched on the device during the last step    */
    float s_norm;        /* ||s_t||_2                                                */
    float r_norm_mean;   /* N_t^-1 sum_{i in I_t} ||r_i||_2; only on steps with an
                            own-step output registered, else 0                      */
    float cancel;        /* within-batch cancellation ratio s_norm / r_norm_mean
                            (drift-measurement appendix), 0 when not measured        */
} bom_stats;

typedef struct bom_handle bom_handle;

/* Parameter tensors, in this order (the grads[] and h_out[] arrays follow the
 * same order and shapes):
 *   for each backbone layer:
 *     LINEAR / LINEAR_GELU : W [d_out, d_in], then b [d_out] if has_bias
 *     SWIGLU               : W_g [ffn, d], W_u [ffn, d], W_d [d, ffn]
 *     RMSNORM              : gamma [d]
 *   head                   : W [d_out, d_model], then b [d_out] if head_bias
 * bom_param_count returns the number of tensors (-1 for a malformed cfg);
 * bom_param_shape the shape of tensor `index`: rows x cols for matrices, and
 * rows = length, cols = 0 for bias vectors. */
int32_t bom_param_count(const bom_config* cfg);
bom_status bom_param_shape(const bom_config* cfg, int32_t index, int64_t* rows, int64_t* cols);

/* Creates a handle: validates cfg, copies it, and allocates the device
 * workspace (activations, logits/residuals, row statistics, column partial
 * sums, scalars) for max_rows rows on the current device.  The handle owns
 * only that workspace.  Returns BOM_EINVAL on a bad config, BOM_ENOTSUP for
 * max_rows above 4,194,240 (64-row blocks of the per-row passes run along
 * one grid dimension of at most 65,535 blocks), on the fp32 path for an
 * output width above the same bound, and for a bf16 width that is not a
 * multiple of 8; BOM_ENOMEM when the workspace does not fit. */
bom_status bom_init(bom_handle** out, const bom_config* cfg);

/* Bytes of device workspace bom_init would allocate for cfg (-1 for a cfg
 * bom_init refuses). */
int64_t bom_workspace_bytes(const bom_config* cfg);

/* One BOM step (Algorithm 1 up to the update numerator).
 *   x       [n_rows, d_in] compute dtype.
 *   labels  [n_rows] int32; ignore_index rows are not supervised.
 *   params  bom_param_count device pointers (compute dtype), read only.
 *   q       [d_out] fp32, in/out: q_{t-1} on entry, q_t on exit (unchanged if
 *           the device latches an error).
 *   t       1-based step index (t >= 1) used by the bias correction; ignored
 *           when a device step counter is registered (bom_set_step_scalars).
 *   grads   bom_param_count output pointers (compute dtype): u, or g in
 *           BOM_OUT_G_AND_H mode.
 *   h_out   BOM_OUT_G_AND_H only: bom_param_count fp32 outputs receiving h;
 *           must be NULL in BOM_OUT_U mode.
 * Requires 1 <= n_rows <= max_rows.  Not re-entrant on one handle: two steps
 * on the same handle must be ordered on one stream. */
bom_status bom_step(bom_handle* h, const void* x, const int32_t* labels, int64_t n_rows,
                    void* const* params, float* q, int64_t t,
                    void* const* grads, void* const* h_out, void* stream);

/* Row-sharded step: the data-parallel split of bom_step at its one exchange
 * (Algorithm 1: s_t is the mean of r_i over the supervised set I_t of the
 * whole batch, and the surrogate's N_t^-1 is the same count; LM construction
 * appendix: ignored targets leave both means).  A batch split by rows over
 * several handles (one per rank, or several on one GPU) computes the step of
 * the whole batch in two calls per shard, with one sum of a small vector
 * between them:
 *
 *   bom_step_shard_begin  forward of this shard's rows, logits, row
 *                         log-sum-exp and residuals R (kept in the handle's
 *                         workspace), then this shard's part of the exchange
 *                         vector xch, fp64 [d_out + 3]:
 *                           xch[j]         sum_{i in I_t^shard} r_ij, j < d_out
 *                           xch[d_out]     sum_{i in I_t^shard} CE_i
 *                           xch[d_out + 1] |I_t^shard| (an integer value)
 *                           xch[d_out + 2] 1 if this shard latched a device
 *                                          error, else 0 (then the sums are 0)
 *                         A shard may hold no supervised row.
 *   the caller            sums the shards' vectors elementwise (one
 *                         all-reduce of d_out + 3 doubles across ranks), so
 *                         that every shard receives the same summed vector;
 *   bom_step_shard_end    from the summed vector: N_t, s_t, the loss,
 *                         q_t = beta1 q_{t-1} + (1-beta1) s_t and qhat_t (every
 *                         shard forms the same q), then the backward of this
 *                         shard's rows with the cotangent
 *                         N_t^-1 [(1-lambda) r_i + lambda qhat_t].  grads[] (and
 *                         h_out[]) receive this shard's share of u (of g and
 *                         h): the shares of all shards sum to the whole
 *                         batch's u, which is the caller's gradient all-reduce
 *                         (the head's rank-1 term uses this shard's
 *                         colsum_{I_t^shard}(H); the head bias share is
 *                         (1-lambda) s^shard + lambda (N_t^shard / N_t) qhat).
 *
 * Both calls take the arguments of bom_step (x, labels, n_rows, params: the
 * same buffers and values in both, unchanged in between); begin takes no q,
 * t or outputs.  One handle per shard; nothing else may run on the handle
 * between the two calls.  begin clears the handle's status word, end keeps
 * it: a device error of begin (bad label, non-finite logits) stops this
 * shard's end, and through xch[d_out + 2] every other shard's end with
 * BOM_ESHARD; a whole batch without supervised rows latches BOM_EEMPTY in
 * every shard.  q (and the device step counter) change only in an end whose
 * status stays clear.  With bom_set_step_scalars, end reads t there and
 * advances it.  Not with the fused update or an own-step output registered
 * (BOM_EINVAL): the update follows the caller's gradient sum.
 *   xch     device fp64 [d_out + 3], 8-byte aligned (BOM_ENOTSUP otherwise);
 *           begin writes it, end reads it. */
bom_status bom_step_shard_begin(bom_handle* h, const void* x, const int32_t* labels, int64_t n_rows,
                                void* const* params, double* xch, void* stream);
bom_status bom_step_shard_end(bom_handle* h, const void* x, const int32_t* labels, int64_t n_rows,
                              void* const* params, float* q, int64_t t, const double* xch,
                              void* const* grads, void* const* h_out, void* stream);

/* Vocabulary-sharded step: the head's output columns (the vocabulary or the
 * classes) split over several handles, every shard with the whole batch and
 * the same backbone.  A row's residual r_ij = exp(z_ij - lse_i) - [j = y_i]
 * (Algorithm 1; Section 3.2) needs the other shards' columns only through the
 * row log-sum-exp lse_i, and s_t, q_t and qhat_t are per column, so they shard
 * with no exchange; the head's input cotangent is a sum over the shards'
 * columns (a R W + b 1_{I_t} (W^T qhat)^T, Eq. mix-gradient).  A step is three
 * calls per shard and two exchanges:
 *
 *   bom_step_vshard_begin  label check and N_t over the whole vocabulary,
 *                          forward, this shard's logits, and its part of each
 *                          row's log-sum-exp:
 *                            lse_part[i] = log sum_{j in shard} exp(z_ij)
 *                          (NaN on every row when this shard latched an
 *                          error);
 *   the caller             gathers every shard's lse_part into
 *                          lse_parts[n_shards, n_rows], in one shard order
 *                          that is the same for every shard (an all-gather);
 *   bom_step_vshard_mid    the row log-sum-exp from the parts (combined in
 *                          that order, so every shard holds the same float),
 *                          R over this shard's columns, s_t, q_t, qhat_t of
 *                          its columns, the head's weight and bias rows of u
 *                          (complete: no other shard adds to them), and this
 *                          shard's part of the head's input cotangent, fp32,
 *                          in dh_part[n_rows, d] (times GELU' of the last
 *                          layer when it is a LINEAR_GELU);
 *   the caller             sums the shards' dh_part elementwise into dh_sum
 *                          (an all-reduce);
 *   bom_step_vshard_end    the backbone's backward from dh_sum: u of every
 *                          backbone tensor, the same on every shard (no
 *                          gradient exchange), and the cotangent of X when an
 *                          input-gradient buffer is registered.
 *
 * The handle's cfg.d_out is this shard's width V_s; its head W [V_s, d] (and
 * bias [V_s]) are rows v_first .. v_first + V_s - 1 of the whole head, and q
 * holds the same V_s entries of the task-space EMA.  Labels are ids of the
 * whole vocabulary [0, v_total) or ignore_index; a supervised row whose label
 * lies outside this shard has no one-hot term here, and counts in N_t like
 * any other.  The three calls take the same x, labels, n_rows and params,
 * unchanged in between, in this order on one stream, and nothing else may run
 * on the handle between them; begin takes no q, t or outputs, end no q or t.
 * grads[] has bom_param_count entries in both mid and end: mid writes the
 * head's, end the backbone's.  bom_get_stats after mid: n_t of the batch, loss
 * = this shard's part of the mean CE (the rows whose label it holds; the
 * shards' parts add up to the loss), s_norm = the norm of this shard's part
 * of s_t.  An error of one shard's begin (a non-finite logit) stops every
 * other shard's mid with BOM_ESHARD through the NaN parts; a bad label or an
 * empty I_t stops every shard (each checks the whole batch).  q changes only
 * in a mid whose status stays clear; with bom_set_step_scalars, mid reads t
 * there and end advances it.  BOM_OUT_U only, and not with the fused update
 * or an own-step output registered (BOM_EINVAL).
 *   v_total    vocabulary size, 1 <= v_total <= INT32_MAX
 *   v_first    this shard's first id, 0 <= v_first <= v_total - cfg.d_out
 *   lse_part   device fp32 [n_rows], 4-byte aligned (BOM_ENOTSUP otherwise)
 *   lse_parts  device fp32 [n_shards, n_rows], 1 <= n_shards <= 4096
 *   dh_part, dh_sum  device fp32 [n_rows, d] (d: the head's input width),
 *              16-byte aligned; needed when the handle has backbone layers or
 *              an input-gradient buffer (NULL allowed otherwise).
 * A mid or end without the matching earlier part (other n_rows, another call
 * in between, an earlier part that failed) returns BOM_EINVAL. */
bom_status bom_step_vshard_begin(bom_handle* h, const void* x, const int32_t* labels, int64_t n_rows,
                                 void* const* params, int64_t v_total, int64_t v_first, float* lse_part,
                                 void* stream);
bom_status bom_step_vshard_mid(bom_handle* h, const void* x, const int32_t* labels, int64_t n_rows,
                               void* const* params, float* q, int64_t t, const float* lse_parts, int32_t n_shards,
                               void* const* grads, float* dh_part, void* stream);
bom_status bom_step_vshard_end(bom_handle* h, const void* x, const int32_t* labels, int64_t n_rows,
                               void* const* params, const float* dh_sum, void* const* grads, void* stream);

/* Fused BOM-AdamW update (Section 3.4; Algorithm 1, last two steps) inside
 * bom_step.  Registers, per parameter tensor, its fp32 master weights theta[k]
 * and fp32 second moment v[k] (shapes as the parameters, 16-byte aligned) and
 * its weight decay wd[k] (host array, copied).  Every following bom_step then
 * applies
 *   v <- beta2 v + (1-beta2) u^2,
 *   theta <- (1 - lr wd) theta - lr u / (sqrt(v / (1-beta2^t)) + eps)
 * to each tensor as soon as its u is complete.  For weight matrices this
 * happens in the epilogue of the GEMM that forms u, which then writes the
 * updated weights in the compute dtype into params[k] instead of writing u.
 * params must therefore be writable, and grads may be NULL (nothing is
 * written there).  Within the step every weight is last read before its
 * update.  The numerator is the fp32 u of the accumulator, not a
 * compute-dtype copy of it.  Requires BOM_OUT_U mode and no own-step output
 * (bom_step returns BOM_EINVAL otherwise).  No update happens in a step whose
 * device status latches an error.  lr usually changes per step: call this
 * again before each step (host-side only), or register a device learning rate
 * with bom_set_step_scalars.  theta = NULL disables it. */
bom_status bom_set_fused_update(bom_handle* h, float* const* theta, float* const* v, const float* wd, float lr,
                                float beta2, float eps);

/* Step scalars on the device, so that one captured step can be replayed for
 * every later step (Algorithm 1 with its bias corrections 1/(1-beta1^t) of q
 * (Section 3.2) and 1/(1-beta2^t) of v (Section 3.4)).
 *   t_dev   int64 device counter (8-byte aligned) holding the index t >= 1 of
 *           the next step.  Every following bom_step reads t there instead of
 *           its t argument (which is then ignored), and increments *t_dev at
 *           its end when it latched no device error, so a failed step leaves
 *           t, like q, unchanged.  A counter below 1 latches BOM_EINVAL.
 *   lr_dev  fp32 device learning rate (4-byte aligned) that the fused update
 *           reads instead of the lr given to bom_set_fused_update, or NULL.
 * The bias corrections computed from *t_dev equal the ones the host forms
 * from the same t (bit for bit), so replayed and directly launched steps give
 * identical results.  Other entry points (bom_update, ...) still take t and
 * lr from the host.  t_dev = NULL and lr_dev = NULL return to host scalars.
 * Returns BOM_ENOTSUP for a misaligned pointer. */
bom_status bom_set_step_scalars(bom_handle* h, int64_t* t_dev, const float* lr_dev);

typedef struct bom_graph bom_graph;

/* Captures one bom_step with these arguments (as bom_step, without t) into an
 * executable CUDA graph, for the small, launch-bound configurations where
 * per-kernel launch cost is a large share of the step.  The graph refers to
 * the given buffers and to the handle's workspace: they must stay allocated,
 * and their contents are read and written at each launch, not at capture.
 * Requires device step scalars (bom_set_step_scalars; BOM_EINVAL otherwise),
 * so each launch runs the step *t_dev and advances the counter.  The settings
 * registered on the handle at capture time (fused update, input gradient,
 * own-step output) are part of the graph; tracing must be off.  The capture
 * runs on a private stream and executes nothing; the handle's first use of a
 * GEMM shape may happen inside it.  Steps of one handle, launched directly or
 * as graphs, must be ordered on one stream. */
bom_status bom_graph_capture(bom_handle* h, const void* x, const int32_t* labels, int64_t n_rows,
                             void* const* params, float* q, void* const* grads, void* const* h_out,
                             bom_graph** out);

/* Launches a captured step on `stream` (asynchronous). */
bom_status bom_graph_launch(bom_graph* g, void* stream);

/* Frees a captured step (NULL is a no-op). */
void bom_graph_destroy(bom_graph* g);

/* Registers a device buffer dx [max_rows, d_in] (compute dtype) that every
 * following bom_step fills with the cotangent of the input X (the u, or in
 * BOM_OUT_G_AND_H mode the g, cotangent): for a head-only configuration
 * this is dH = N_t^-1 [(1-lambda) R W + lambda 1_{I_t} (W^T qhat)^T], the
 * input-side half of the head backward.  NULL disables it (the default). */
bom_status bom_set_input_grad(bom_handle* h, void* dx);

/* Drift telemetry and the own-step control (Section 3.3, Eq. drift-telemetry;
 * stale-control and drift-measurement appendices).
 * Registers bom_param_count fp32 device buffers (shapes as the parameters)
 * that every following bom_step fills with the own-step projection
 * o_t = Jbar_t^T s_t: one extra backward of the logit cotangent
 * N_t^-1 1_{I_t} s_t^T through the current model and batch.  Such steps also
 * measure the per-row residual norms for bom_stats.r_norm_mean / cancel.
 * NULL disables it (the default).  Returns BOM_ENOTSUP for a buffer that is
 * not 16-byte aligned. */
bom_status bom_set_own_step_output(bom_handle* h, void* const* o);

/* Own-step moment over a flat range of n fp32 elements:
 *   M <- beta1 M + (1 - beta1) o,   mhat = M / (1 - beta1^t)
 * (M_0 = 0; the own-step control then updates with u = (1-lambda) g +
 * lambda mhat, i.e. bom_update with hvec = mhat).  When sums is non-NULL,
 * hvec ([n] fp32: h_t = Jbar_t^T qhat_t of the same step) must be given and
 *   sums[0..3] += ( <mhat,h>, <mhat,mhat>, <h,h>, <mhat-h,mhat-h> )
 * in fp64 and a fixed summation order, from which cos(Mhat_t, h_t) and
 * ||Mhat_t - h_t|| / ||Mhat_t|| follow; calling it per tensor range with one
 * sums buffer per group (e.g. head, encoder) gives the paper's split.
 * M, o, hvec, mhat: device fp32 [n], 16-byte aligned (else BOM_ENOTSUP);
 * sums: device fp64 [4] or NULL.
 * Uses a per-handle partials buffer: calls on one handle must be ordered on
 * one stream.  Asynchronous; t >= 1 and 0 <= beta1 < 1 or BOM_EINVAL. */
bom_status bom_own_step_moment(bom_handle* h, float* M, const float* o, const float* hvec, float* mhat,
                               int64_t n, float beta1, int64_t t, double* sums, void* stream);

/* Bytes bom_get_stats copies from the device per call. */
int64_t bom_stats_transfer_bytes(void);

/* Device-side outputs of the last step that are useful for checks:
 *   qhat [d_out] fp32, s [d_out] fp32, lse [n_rows] fp32 (row log-sum-exp).
 * Pointers stay valid until bom_destroy; contents until the next bom_step. */
bom_status bom_step_outputs(bom_handle* h, const float** qhat, const float** s, const float** lse);

/* Synchronises `stream` and copies the statistics of the last step.  Returns
 * the latched device status (BOM_OK when the step succeeded). */
bom_status bom_get_stats(bom_handle* h, bom_stats* out, void* stream);

/* The same statistics without a synchronisation: enqueues on `stream`, after
 * the work already there, a copy of bom_stats_transfer_bytes() bytes of the
 * device statistics block into host memory `dst` (caller-owned; page-locked
 * for the copy to be asynchronous), and returns.  Once the stream has passed
 * that point (an event recorded after the call, say), bom_stats_decode(dst,
 * out) fills `out` and returns the latched status, as bom_get_stats does.
 * A later step on the handle overwrites the device block, not `dst`: a
 * caller that keeps one step in flight reads step t's statistics while step
 * t + 1 runs (the loss read-back of a training loop).  BOM_EINVAL for NULL
 * h or dst, BOM_ECUDA when the copy cannot be enqueued. */
bom_status bom_get_stats_async(bom_handle* h, void* dst, void* stream);
bom_status bom_stats_decode(const void* src, bom_stats* out);

/* BOM-AdamW update over a flat range of n elements (Section 3.4).
 *   theta       [n] fp32 master parameters, updated in place.
 *   g           [n] in g_dtype (BOM_F32 or BOM_BF16): u itself when hvec is
 *               NULL, otherwise the supervised gradient g and the kernel forms
 *               u = (1-lambda) g + lambda hvec (Eq. mix-gradient).
 *   hvec        [n] fp32 reprojection h, or NULL.
 *   v           [n] fp32 second moment, updated in place (v_0 = 0).
 *   theta_bf16  [n] optional bf16 copy of the updated theta (NULL: none).
 *   lr, wd      eta_t and the decoupled weight-decay coefficient omega.
 *   t           1-based step index.
 * All pointers 16-byte aligned.  n = 0 is a no-op. */
bom_status bom_update(float* theta, const void* g, int32_t g_dtype, const float* hvec, float* v,
                      uint16_t* theta_bf16, int64_t n, float lr, float wd, float lambda,
                      float beta2, float eps, int64_t t, void* stream);

/* BOM-Adam-mini update (Section 3.5, composition with Adam-mini; the
 * optimizer-implementation appendix): as bom_update, but one second-moment
 * scalar is shared by each block of `block` consecutive elements,
 *   v_b  <- beta2 v_b + (1-beta2) mean_{i in b} u_i^2,
 *   theta <- (1 - lr wd) theta - lr u / (sqrt(v_b / (1-beta2^t)) + eps).
 * A row-major [d_out, d_in] weight with block = d_in shares v per output
 * neuron, block = n shares it over the whole tensor, block = 1 is bom_update;
 * the last block may be shorter.
 *   v_blocks    [ceil(n / block)] fp32, updated in place (v_0 = 0).
 * Other arguments as bom_update.  block >= 1; sums of u^2 are formed per
 * block in a fixed order (deterministic).  Blocks of more than 8192 elements,
 * when there are fewer of them than the GPU runs 8-CTA clusters at once, are
 * spread over the whole grid: that path takes a few KB of stream-ordered
 * scratch from a memory pool the library keeps per device (BOM_ENOMEM if it
 * cannot). */
/* Global-norm clipping of the numerator (pretraining-parameters appendix:
 * language-modeling runs clip at 1.0; convergence appendix: the clipped
 * numerator is what the adaptive update receives).  Two calls:
 *   bom_sqnorm          *sq += sum u_i^2 over a flat range (u = g, or
 *                       (1-lambda) g + lambda hvec when hvec is given), in fp64
 *                       and a fixed order; call it for every range of the
 *                       clipping group into one zeroed device double;
 *   bom_update_clipped  bom_update with u scaled first by
 *                       c = min(1, max_norm / (sqrt(*sq) + 1e-6)).
 * bom_sqnorm uses the handle's partials buffer: calls on one handle must be
 * ordered on one stream.  max_norm > 0; other arguments as bom_update. */
bom_status bom_sqnorm(bom_handle* h, const void* g, int32_t g_dtype, const float* hvec, float lambda, int64_t n,
                      double* sq, void* stream);
bom_status bom_update_clipped(float* theta, const void* g, int32_t g_dtype, const float* hvec, float* v,
                              uint16_t* theta_bf16, int64_t n, float lr, float wd, float lambda, float beta2,
                              float eps, int64_t t, const double* sq, float max_norm, void* stream);

bom_status bom_update_blockshared(float* theta, const void* g, int32_t g_dtype, const float* hvec, float* v_blocks,
                                  uint16_t* theta_bf16, int64_t n, int64_t block, float lr, float wd, float lambda,
                                  float beta2, float eps, int64_t t, void* stream);

/* Auxiliary: D = alpha * op(A) op(B)^T on the bf16 tensor-core GEMM engine the
 * step uses (tcgen05 MMA, TMEM accumulators, TMA loads), fp32 accumulation,
 * fp32 output D [M, N] with row pitch ldd.  A is M x K: a_mn_major = 0 means
 * element (m,k) is at A[m*lda + k], 1 means at A[k*lda + m]; B likewise for
 * N x K.  Exposed so the engine can be tested on its own. */
bom_status bom_gemm_bf16(const uint16_t* A, int64_t lda, int32_t a_mn_major,
                         const uint16_t* B, int64_t ldb, int32_t b_mn_major,
                         float* D, int64_t ldd, int64_t M, int64_t N, int64_t K,
                         float alpha, void* stream);

/* Tracing (the measurement support of the step; the paper times whole steps
 * with CUDA events, Appendix measurement-protocol).  While enabled on a
 * handle, bom_step records a CUDA event pair on `stream` around every kernel
 * it launches, with the algorithmic FLOPs and HBM bytes of that launch.
 * bom_trace(h, 1) enables and clears the record, bom_trace(h, 0) disables. */
typedef struct {
    const char* name;   /* kernel class, e.g. "gemm_tc.logits" (static string)   */
    double flops;       /* algorithmic floating-point operations of the launch   */
    double bytes;       /* algorithmic HBM bytes of the launch                   */
    float ms;           /* device time between the event pair                    */
} bom_trace_entry;
bom_status bom_trace(bom_handle* h, int32_t enable);

/* Synchronises `stream`, then copies up to `max` entries of the launches of
 * the most recent bom_step into `out`; returns how many the step recorded
 * (or -1 on error). */
int32_t bom_trace_read(bom_handle* h, bom_trace_entry* out, int32_t max, void* stream);

/* Number of kernels this library has launched in the process so far (a
 * captured step counts its kernels each time it is launched, not when it is
 * captured). */
int64_t bom_launch_count(void);

/* Allocation-free weighted column sum (the paper has no counterpart; this is
 * a convenience of this library).
 *   out[j] = sum_i w_i * x[i, j]   for j < n_cols, with w_i = weights[i], or 1
 *   when weights is NULL; fp32 accumulation, fp32 out [n_cols].
 * This is the reduction bom_step uses to form colsum_{I_t}(H) and W^T qhat,
 * for callers that may not allocate device memory: code running while its
 * stream is being captured into a CUDA graph in global capture mode, where
 * cudaMalloc is an error, and runtimes that manage every device byte through
 * their own pool.  It calls no cudaMalloc/cudaFree and no allocating library
 * routine.  Its scratch is one fixed device array of 4 MiB (2^20 floats) in
 * the library; every GPU that loads the library keeps it until exit.
 *   x        [n_rows, ldx] in dtype (BOM_F32 or BOM_BF16), 16-byte aligned.
 *   weights  [n_rows] fp32 device vector, or NULL.
 *   out      [n_cols] fp32 device vector.
 * Limits: ceil(n_rows / 128) * n_cols <= 2^20 and n_rows <= 128 * 65535;
 * larger sizes return BOM_ENOTSUP without touching the device.
 * The first call on each device looks up the array's device address with
 * cudaGetSymbolAddress; make that first call before any stream capture.
 * All calls share the array: calls that overlap on the GPU (on different
 * streams without ordering) race and produce wrong sums.  Each call writes
 * every scratch element it later reads, so nothing needs to start at zero. */
bom_status bom_colsum_noalloc(const void* x, int32_t dtype, int64_t ldx, int64_t n_rows, int64_t n_cols,
                              const float* weights, float* out, void* stream);

/* Frees the workspace and the handle.  NULL is a no-op. */
void bom_destroy(bom_handle* h);

/* Static string naming a status code. */
const char* bom_status_string(bom_status s);

#ifdef __cplusplus
}
#endif

#endif /* BOM_H */
