// Launchers of the non-GEMM kernels of the BOM step and of the update.
#pragma once
#include <cstdint>
#include <cuda_runtime.h>

#include "common.cuh"

namespace bom {

// Row-block height that sizes the partial-sum buffers of the column
// reductions (they use row ranges of at least this many rows).  The column
// partial sums of one block are summed in a fixed order afterwards, so every
// reduction of the step is deterministic (no float atomics).
constexpr int kRowBlock = 128;

// Streaming multiprocessors of the current device (cached on first use).
int device_sm_count();

inline int64_t row_blocks(int64_t n) { return (n + kRowBlock - 1) / kRowBlock; }

// Row-block height of the residual pass (its column partial sums feed s_t).
constexpr int kResidRows = 64;
inline int64_t resid_blocks(int64_t n) { return (n + kResidRows - 1) / kResidRows; }

// Counts N_t, checks every label, latches BOM_ELABEL / BOM_EEMPTY and writes
// the cotangent coefficients of the four backward passes into sc.
// Where the step scalars (lr, 1/(1 - beta1^t), 1/(1 - beta2^t)) of a step come
// from: the host values here, or the device step counter t_dev (and the device
// learning rate lr_dev) registered with bom_set_step_scalars.  The label scan
// writes them into sc; a t_dev below 1 latches BOM_EINVAL.
struct StepScalarsIn {
    float lr, inv_bc1, inv_bc2;
    const int64_t* t_dev;
    const float* lr_dev;
    float beta1, beta2;
};
// allow_empty (the first half of a row-sharded step): N_t = 0 is not an error.
void launch_labels_scan(const int32_t* labels, int64_t n, int64_t V, int32_t ignore, float lambda,
                        const StepScalarsIn& st, DevScalars* sc, cudaStream_t s, bool allow_empty = false);

// *t_dev += 1 when the step latched no error (the last kernel of a step that
// reads its t from the device).
void launch_advance_step(int64_t* t_dev, const DevScalars* sc, cudaStream_t s);

// fp32 path: per-row (max, sum exp) of Z [n, ldz] over V columns (one tile).
void launch_row_stats_f32(const float* Z, int64_t ldz, int64_t n, int64_t V, float* stats, const DevScalars* sc,
                          cudaStream_t s);

// Merges per-tile (max, sum exp) pairs into lse[i]; ce[i] = lse_i - z_{i,y_i}
// for supervised rows, 0 otherwise.
void launch_row_lse(const void* Z, int z_f32, int64_t ldz, int64_t n, int64_t V, const float* stats, int64_t ntiles,
                    const int32_t* labels, int32_t ignore, float* lse, float* ce, DevScalars* sc,
                    cudaStream_t s);

// Z -> R in place: r_ij = exp(z_ij - lse_i) - [j = y_i] on supervised rows, 0 on
// the others and in the padding columns [V, ldz); colpart[b, j] receives the
// fp32 column sums of r over row block b.
// yoff: the label of column j is yoff + j (a vocabulary shard's first id; 0 otherwise).
void launch_residual(void* Z, int z_f32, int64_t ldz, int64_t n, int64_t V, const float* lse, const int32_t* labels,
                     int32_t ignore, float* colpart, const DevScalars* sc, cudaStream_t s, int64_t yoff = 0);

// s_j = N_t^-1 sum_b colpart[b, j]; q_j <- beta1 q_j + (1-beta1) s_j;
// qhat_j = q_j * inv_bc1.  q is only written when the status word is clear.
void launch_finish_sq(const float* colpart, int64_t nblocks, int64_t V, float beta1, float* q,
                      float* s_out, float* qhat, DevScalars* sc, cudaStream_t s);

// Row-sharded step (see bom_step_shard_begin / _end in bom.h).
// xch[0, V) = fixed-order column sums of colpart, xch[V] = sum_i ce_i,
// xch[V+1] = this shard's N_t, xch[V+2] = 1 if the status word is set.
void launch_shard_sums(const float* colpart, int64_t nblocks, const float* ce, int64_t n, int64_t V, double* xch,
                       const DevScalars* sc, cudaStream_t s);
// From the summed xch: N_t, 1/N_t, cotangent coefficients, loss, step scalars,
// shard_frac; latches BOM_ESHARD / BOM_EEMPTY.
void launch_shard_scalars_in(const double* xch, int64_t V, float lambda, const StepScalarsIn& st, DevScalars* sc,
                             cudaStream_t s);
// s = xch / N_t, q EMA, qhat, and s_shard = (this shard's column sums) / N_t.
void launch_shard_finish_sq(const double* xch, const float* colpart, int64_t nblocks, int64_t V, float beta1,
                            float* q, float* s_out, float* qhat, float* s_shard, const DevScalars* sc,
                            cudaStream_t s);
// out[j] = a s_shard[j] + b shard_frac qhat[j] (this shard's head bias share).
void launch_shard_bias(const float* s_shard, const float* qhat, float a, float b, int64_t V, void* out, int out_f32,
                       const DevScalars* sc, cudaStream_t s);

// Vocabulary-sharded step (see bom_step_vshard_begin / _mid / _end in bom.h).
// lse_part[i] = log sum over this shard's columns of exp(z_ij), from the
// per-tile statistics (NaN on every row when the status word is set).
void launch_vshard_lse_part(const float* stats, int64_t ntiles, int64_t n, float* lse_part, DevScalars* sc,
                            cudaStream_t s);
// lse[i] from the shards' parts [nsh, n] in shard order, ce[i] on the rows whose
// label lies in [v0, v0 + Vloc), the step scalars; BOM_ESHARD on a NaN part.
void launch_vshard_lse(const float* parts, int32_t nsh, int64_t n, const void* Z, int z_f32, int64_t ldz, int64_t v0,
                       int64_t Vloc, const int32_t* labels, int32_t ignore, float* lse, float* ce,
                       const StepScalarsIn& st, DevScalars* sc, cudaStream_t s);
// dst[0, n) = src (bf16 round to nearest, or fp32); 16-byte aligned buffers.
void launch_cast_f32(const float* src, void* dst, int64_t n, int dst_f32, const DevScalars* sc, cudaStream_t s);

// Task-space pass of a small step in one cluster launch (task_small.cu):
// label check and N_t, row log-sum-exp and CE, R over Z, s_t, q_t, qhat_t,
// the step scalars, c = colsum_{I_t}(H) (H [n, dm]), w = W^T qhat (W [V, dm])
// and, when hb_out is given, the head bias numerator hb_a s + hb_b qhat.  Used
// for n <= 4096 rows, V and dm <= 8192 and n V <= 2^19 when a cluster of 8
// CTAs fits on the device (task_small_usable).
constexpr int64_t kTaskSmallMaxRows = 4096;
constexpr int64_t kTaskSmallMaxV = 8192;
constexpr int64_t kTaskSmallMaxD = 8192;
constexpr int64_t kTaskSmallMaxElems = int64_t(1) << 19;
bool task_small_usable(int64_t n, int64_t V, int64_t dm, int z_f32);
int launch_task_small(const void* Z, int z_f32, int64_t ldz, const int32_t* labels, int64_t n, int64_t V,
                      int32_t ignore, float lambda, float beta1, const void* H, const void* W, int64_t dm, float* q,
                      float* s_out, float* qhat, float* lse, float* cvec, float* wvec, void* hb_out, int hb_f32,
                      float hb_a, float hb_b, const StepScalarsIn& st, DevScalars* sc, cudaStream_t s);

// Whole step of a small fp32 MLP classifier (at most two Linear / Linear+GELU
// layers before the head, at most 128 rows, widths at most 1024, everything in
// 192 KB of shared memory) in one CTA (tiny_step.cu): forward, task space,
// backward and either the fused update or u.  The layout holds the
// shared-memory offsets (floats) of the staged operands and intermediates.
constexpr int kTinyStepMaxLayers = 2;
constexpr int kTinyStepMaxRows = 128;
constexpr int kTinyStepMaxWidth = 1024;
constexpr int64_t kTinyStepMaxFloats = 48 * 1024;
struct TinyLayout {
    int x, W[kTinyStepMaxLayers + 1], b[kTinyStepMaxLayers + 1], pre[kTinyStepMaxLayers], act[kTinyStepMaxLayers];
    int z, g[2], lse, lab, qh, sv, floats;
};
struct TinyStepArgs {
    const float* x;                              // [n, dim[0]]
    const int32_t* labels;                       // [n]
    int n, nl;                                   // rows, backbone layers
    int dim[kTinyStepMaxLayers + 2];             // input width, layer widths, classes
    int gelu[kTinyStepMaxLayers];                // layer k applies GELU
    const float* W[kTinyStepMaxLayers + 1];      // layer weights [dim[k+1], dim[k]]; the head last
    const float* b[kTinyStepMaxLayers + 1];      // biases, or null
    int tw[kTinyStepMaxLayers + 1];              // tensor index of W[k] (parameter order)
    int tb[kTinyStepMaxLayers + 1];              // tensor index of b[k], or -1
    int32_t ignore;
    float lambda, beta1;
    float* q;                                    // [V] in/out
    float *qhat_out, *s_out, *lse_out;           // the handle's outputs
    float* u[2 * kTinyStepMaxLayers + 2];        // u per tensor (when theta is null)
    float* theta[2 * kTinyStepMaxLayers + 2];    // fused update: fp32 masters, or null
    float* v[2 * kTinyStepMaxLayers + 2];
    float wd[2 * kTinyStepMaxLayers + 2];
    float* copy[2 * kTinyStepMaxLayers + 2];     // compute copies (the parameters)
    float beta2, eps;
    StepScalarsIn st;
    DevScalars* sc;
    int64_t* t_adv;                              // device step counter advanced when clear, or null
    TinyLayout lay;
};
bool tiny_step_layout(int n, int nl, const int* dim, const bool* bias, TinyLayout* lay);
int launch_tiny_step(const TinyStepArgs& a, cudaStream_t s);

// loss = N_t^-1 sum_i ce_i (kept as it is when ce is NULL), ||s|| and, when
// rnorm is given, r_norm_mean = N_t^-1 sum_i rnorm_i.
void launch_scalars(const float* ce, int64_t n, const float* s_vec, int64_t V, const float* rnorm, DevScalars* sc,
                    cudaStream_t s);

// rnorm[i] = ||R[i, 0:V]||_2 (one warp per row).
void launch_row_norm(const void* R, int r_f32, int64_t ldr, int64_t n, int64_t V, float* rnorm, const DevScalars* sc,
                     cudaStream_t s);

// Grid of the own-step moment pass for n elements on a device with `sms` SMs;
// the pass needs 4 * own_step_blocks(n) doubles of partials.
constexpr int kOwnStepMaxBlocks = 1024;
int own_step_blocks(int64_t n, int sms);

// M <- beta1 M + (1-beta1) o; mhat = M * inv_bc1; when sums is given (and hv),
// sums[0..3] += (<mhat,hv>, <mhat,mhat>, <hv,hv>, <mhat-hv,mhat-hv>) in a fixed order.
void launch_own_step_moment(float* M, const float* o, const float* hv, float* mhat, int64_t n, float beta1,
                            float inv_bc1, double* part, int nblocks, double* sums, cudaStream_t s);

// out[j] = scale * sum_i w_i X[i, j]  (w_i = 1, the row mask from labels, or wvec[i]).
// `part` must hold row_blocks(n) * d floats.
void launch_colsum(const void* X, int x_f32, int64_t ldx, int64_t n, int64_t d, const int32_t* labels,
                   int32_t ignore, const float* wvec, float scale, float* part, void* out, int out_f32,
                   const DevScalars* sc, cudaStream_t s);

// As launch_colsum with an elementwise second factor: out[j] = scale * sum_i w_i X[i, j] Y[i, j]
// (Y has X's layout; Y = NULL is launch_colsum).
void launch_colsum2(const void* X, const void* Y, int x_f32, int64_t ldx, int64_t n, int64_t d,
                    const int32_t* labels, int32_t ignore, const float* wvec, float scale, float* part, void* out,
                    int out_f32, const DevScalars* sc, cudaStream_t s);

// RMSNorm (norm.cu): rstd[i] = 1 / sqrt(mean_j x_ij^2 + 1e-6), y = x rstd gamma.
void launch_rmsnorm_fwd(const void* x, const void* gamma, void* y, float* rstd, int64_t n, int64_t d, int f32,
                        const DevScalars* sc, cudaStream_t s);
// dx = rstd (dy gamma - xhat mean_j(dy gamma xhat)), times GELU'(pre) when pre is given.
void launch_rmsnorm_bwd(const void* dy, const void* x, const void* gamma, const float* rstd, const void* pre,
                        void* dx, int64_t n, int64_t d, int f32, const DevScalars* sc, cudaStream_t s);

// out[j] = a * s[j] + b * qhat[j] (head bias numerator).
void launch_axpby(const float* s_vec, const float* qhat, float a, float b, int64_t V, void* out, int out_f32,
                  const DevScalars* sc, cudaStream_t s);

// BOM-Adam-mini update with one second moment per block (see bom_update_blockshared in bom.h).
int launch_update_blockshared(float* theta, const void* g, int g_bf16, const float* h, float* vb, uint16_t* shadow,
                              int64_t n, int64_t block, float lr, float wd, float lambda, float beta2, float eps,
                              float inv_bc2, cudaStream_t s);

// BOM-AdamW update (see bom_update in bom.h).  With clip_sq, u is first scaled
// by min(1, max_norm / (sqrt(*clip_sq) + 1e-6)) (bom_update_clipped).
// When sc is given the kernel does nothing once the step's status word is set.
// With step_scalars, lr and inv_bc2 are taken from sc's step scalars instead
// (the vector updates inside bom_step).
int launch_update(float* theta, const void* g, int g_bf16, const float* h, float* v, uint16_t* shadow, int64_t n,
                  float lr, float wd, float lambda, float beta2, float eps, float inv_bc2, const double* clip_sq,
                  float max_norm, const DevScalars* sc, cudaStream_t s, bool step_scalars = false);

// BOM-AdamW update of up to kMultiUpdMax tensors in one launch: fp32 theta,
// v and u (16-byte aligned) and the compute copy of each (bf16, or fp32 when
// copy_f32); lr and 1/(1 - beta2^t) from the step scalars in sc; nothing when
// sc's status is set.  A tensor k with src[k] given is a bias whose u is the
// column sum of src[k] [rows[k], n[k]] (rows in order; fp32 when src_f32[k]
// is 1, else the compute dtype; src_f32 null: the compute dtype).  t_adv
// (or null): a device step counter advanced by one when sc's status is clear.
constexpr int kMultiUpdMax = 24;
int launch_update_multi(int ntensor, float* const* theta, float* const* v, const float* const* u, void* const* copy,
                        int copy_f32, const int64_t* n, const float* wd, const void* const* src, const int64_t* rows,
                        const int* src_f32, float beta2, float eps, const DevScalars* sc, int64_t* t_adv,
                        cudaStream_t s);

// *sq += sum u^2 over n elements (u = g, or (1-lambda) g + lambda h), in a fixed
// order; `part` holds kOwnStepMaxBlocks doubles.
int launch_sqnorm(const void* g, int g_bf16, const float* h, float lambda, int64_t n, double* part, double* sq,
                  cudaStream_t s);

}  // namespace bom
