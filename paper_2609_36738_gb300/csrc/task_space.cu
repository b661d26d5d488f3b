// Task-space part of the BOM step (Algorithm 1, residual / EMA steps):
// label scan and N_t, row log-sum-exp from the logits epilogue's per-tile
// statistics, the residual pass r = softmax(z) - onehot(y) with deterministic
// column partial sums, s_t and the q_t EMA with bias correction, and the
// column reductions colsum_{I_t}(H), W^T qhat and bias gradients.
#include <algorithm>

#include "kernels.h"

namespace bom {

namespace {

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    return v;
}
__device__ __forceinline__ float warp_max(float v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
    return v;
}
__device__ __forceinline__ int warp_sum_i(int v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    return v;
}

// Sum over the nblocks rows of part[nblocks, ncols] for 32 consecutive columns
// per 256-thread block: warp w adds rows w, w+8, ..., then warp 0 adds the 8
// warp sums in order.  Fixed order for fixed sizes (deterministic); the result
// is valid in warp 0 (lane l holds column `col` of lane l).
__device__ __forceinline__ float fixed_order_column_sum(const float* __restrict__ part, int64_t nblocks,
                                                        int64_t ncols, int64_t col, float (*red)[33]) {
    const int w = threadIdx.x >> 5, l = threadIdx.x & 31;
    // eight independent loads in flight per thread: the pass is latency-bound
    float a[8];
#pragma unroll
    for (int k = 0; k < 8; ++k) a[k] = 0.0f;
    if (col < ncols) {
        int64_t b = w;
        for (; b + 56 < nblocks; b += 64) {
#pragma unroll
            for (int k = 0; k < 8; ++k) a[k] += part[(b + 8 * k) * ncols + col];
        }
        for (; b < nblocks; b += 8) a[0] += part[b * ncols + col];
    }
    red[w][l] = ((a[0] + a[1]) + (a[2] + a[3])) + ((a[4] + a[5]) + (a[6] + a[7]));
    __syncthreads();
    float r = 0.0f;
    if (w == 0) {
#pragma unroll
        for (int k = 0; k < 8; ++k) r += red[k][l];
    }
    return r;
}

// Deterministic block sum of a float (fixed tree for a fixed block size).
template <int NT>
__device__ float block_sum(float v, float* red) {
    v = warp_sum(v);
    const int w = threadIdx.x >> 5, l = threadIdx.x & 31;
    if (l == 0) red[w] = v;
    __syncthreads();
    float r = 0.0f;
    if (w == 0) {
        r = (l < NT / 32) ? red[l] : 0.0f;
        r = warp_sum(r);
    }
    __syncthreads();
    return r;  // valid in thread 0
}

// The step counter advances only after a step that latched no error, so a
// failed step leaves t, like q, as it was.
__global__ void advance_step_kernel(int64_t* __restrict__ t, const DevScalars* sc) {
    pdl_enter();
    if (threadIdx.x == 0 && sc->status == 0) *t += 1;
}

// allow_empty: a row shard of a sharded step may hold no supervised row; only
// the whole batch's N_t must be positive (checked when the shards' sums meet).
__global__ void labels_scan_kernel(const int32_t* __restrict__ labels, int64_t n, int64_t V, int32_t ignore,
                                   float lambda, const StepScalarsIn st, int allow_empty, DevScalars* sc) {
    pdl_enter();
    __shared__ int s_cnt[32], s_bad[32];
    int cnt = 0, bad = 0;
    for (int64_t i = threadIdx.x; i < n; i += blockDim.x) {
        const int32_t y = labels[i];
        if (y == ignore) continue;
        if (y < 0 || y >= V)
            ++bad;
        else
            ++cnt;
    }
    cnt = warp_sum_i(cnt);
    bad = warp_sum_i(bad);
    const int w = threadIdx.x >> 5, l = threadIdx.x & 31;
    if (l == 0) {
        s_cnt[w] = cnt;
        s_bad[w] = bad;
    }
    __syncthreads();
    if (threadIdx.x == 0) {
        int c = 0, b = 0;
        for (int k = 0; k < (int)(blockDim.x >> 5); ++k) {
            c += s_cnt[k];
            b += s_bad[k];
        }
        sc->n_t = c;
        if (b > 0)
            latch_status(sc, BOM_ELABEL);
        else if (c == 0 && !allow_empty)
            latch_status(sc, BOM_EEMPTY);
        const float inv = c > 0 ? 1.0f / static_cast<float>(c) : 0.0f;
        sc->inv_nt = inv;
        sc->coef_r[0] = (1.0f - lambda) * inv;  // u pass: N_t^-1 (1-lambda) r_i
        sc->coef_q[0] = lambda * inv;           //         N_t^-1 lambda qhat
        sc->coef_r[1] = inv;                    // g pass: N_t^-1 r_i
        sc->coef_q[1] = 0.0f;
        sc->coef_r[2] = 0.0f;                   // h pass: N_t^-1 qhat
        sc->coef_q[2] = inv;
        sc->coef_r[3] = 0.0f;                   // own-step pass: N_t^-1 s_t
        sc->coef_q[3] = inv;
        float bc1 = st.inv_bc1, bc2 = st.inv_bc2;
        if (st.t_dev != nullptr) {
            const int64_t t = *st.t_dev;
            if (t < 1) {
                latch_status(sc, BOM_EINVAL);
            } else {
                bc1 = inv_bias_correction(st.beta1, t);
                bc2 = inv_bias_correction(st.beta2, t);
            }
        }
        sc->lr = st.lr_dev != nullptr ? *st.lr_dev : st.lr;
        sc->inv_bc1 = bc1;
        sc->inv_bc2 = bc2;
        sc->loss = 0.0f;
        sc->s_norm = 0.0f;
        sc->r_norm_mean = 0.0f;
    }
}

// One warp per row.
__global__ void row_stats_f32_kernel(const float* __restrict__ Z, int64_t ldz, int64_t n, int64_t V,
                                     float2* __restrict__ stats, const DevScalars* sc) {
    pdl_enter();
    if (sc->status != 0) return;
    const int64_t row = (static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x) >> 5;
    const int l = threadIdx.x & 31;
    if (row >= n) return;
    const float* z = Z + row * ldz;
    float m = -INFINITY;
    for (int64_t j = l; j < V; j += 32) m = fmaxf(m, z[j]);
    m = warp_max(m);
    float s = 0.0f;
    for (int64_t j = l; j < V; j += 32) s += expf(z[j] - m);
    s = warp_sum(s);
    if (l == 0) stats[row] = make_float2(m, s);
}

__global__ void row_lse_kernel(const void* __restrict__ Z, int z_f32, int64_t ldz, int64_t n, int64_t V,
                               const float2* __restrict__ stats, int64_t ntiles, const int32_t* __restrict__ labels,
                               int32_t ignore, float* __restrict__ lse, float* __restrict__ ce, DevScalars* sc) {
    pdl_enter();
    if (sc->status != 0) return;
    const int64_t row = (static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x) >> 5;
    const int l = threadIdx.x & 31;
    if (row >= n) return;
    const int32_t y = labels[row];
    const float2* st = stats + row * ntiles;
    // the first 256 (max, sum) pairs of the row stay in registers: one read
    // with eight loads in flight per lane (a row of the 32000-column head has
    // 250); pairs beyond are read again for the sum
    constexpr int kRegPairs = 8;
    float2 v[kRegPairs];
#pragma unroll
    for (int k = 0; k < kRegPairs; ++k) {
        const int64_t t = l + 32 * k;
        v[k] = t < ntiles ? st[t] : make_float2(-INFINITY, 0.0f);
    }
    float zy = 0.0f;
    const bool has_y = y != ignore && y >= 0 && y < V;
    if (l == 0 && has_y) zy = ld_elem(Z, row * ldz + y, z_f32);
    float m = -INFINITY;
#pragma unroll
    for (int k = 0; k < kRegPairs; ++k) m = fmaxf(m, v[k].x);
    for (int64_t t = l + 32 * kRegPairs; t < ntiles; t += 32) m = fmaxf(m, st[t].x);
    m = warp_max(m);
    float s = 0.0f;
#pragma unroll
    for (int k = 0; k < kRegPairs; ++k)
        if (v[k].x != -INFINITY) s += v[k].y * expf(v[k].x - m);
    for (int64_t t = l + 32 * kRegPairs; t < ntiles; t += 32) {
        const float2 p = st[t];
        if (p.x != -INFINITY) s += p.y * expf(p.x - m);
    }
    s = warp_sum(s);
    if (l == 0) {
        const float L = m + logf(s);
        lse[row] = L;
        ce[row] = has_y ? L - zy : 0.0f;
        // a non-finite row (ignored or not: its activations still reach the
        // weight gradients) stops the step before q or any parameter changes
        if (!isfinite(L) || (has_y && !isfinite(zy))) latch_status(sc, BOM_ENONFINITE);
    }
}

// Block: 256 threads x VEC consecutive columns (one 16-byte word each) of
// kResidRows rows.  The words of UNROLL rows are loaded before any is used and
// stay packed until then, so a thread keeps 128 bytes in flight with few
// registers and three blocks fit on an SM.  The pass is issue-bound as much as
// HBM-bound, so the bf16 form works on value pairs (paired fma / add, one
// exponential per value), decides row validity once per row and subtracts the
// one-hot only in the thread whose columns hold the label.
template <typename T, int VEC>
__global__ void __launch_bounds__(256, 3) residual_kernel(T* __restrict__ Z, int64_t ldz, int64_t n, int64_t V,
                                                          const float* __restrict__ lse,
                                                          const int32_t* __restrict__ labels, int32_t ignore,
                                                          int64_t yoff, float* __restrict__ colpart,
                                                          const DevScalars* sc) {
    pdl_enter();
    if (sc->status != 0) return;
    const int64_t col0 = (static_cast<int64_t>(blockIdx.x) * 256 + threadIdx.x) * VEC;
    const int64_t r0 = static_cast<int64_t>(blockIdx.y) * kResidRows;
    const int64_t r1 = min(r0 + kResidRows, n);
    if (col0 >= ldz) return;
    constexpr int UNROLL = 8;
    if constexpr (sizeof(T) == 2) {
        static_assert(VEC == 8, "bf16 rows are handled as 16-byte words");
        const bool full = col0 + VEC <= V;
        float2 cs[4];
#pragma unroll
        for (int k = 0; k < 4; ++k) cs[k] = make_float2(0.0f, 0.0f);
        const float2 l2 = make_float2(kLog2e, kLog2e);
        for (int64_t rb = r0; rb < r1; rb += UNROLL) {
            uint4 raw[UNROLL];
#pragma unroll
            for (int u = 0; u < UNROLL; ++u)
                if (rb + u < r1) raw[u] = *reinterpret_cast<const uint4*>(Z + (rb + u) * ldz + col0);
#pragma unroll
            for (int u = 0; u < UNROLL; ++u) {
                const int64_t r = rb + u;
                if (r >= r1) break;
                uint4* dst = reinterpret_cast<uint4*>(Z + r * ldz + col0);
                const int32_t y = labels[r];
                if (y == ignore) {   // ignored rows contribute nothing
                    *dst = make_uint4(0u, 0u, 0u, 0u);
                    continue;
                }
                const float Ls = lse[r] * kLog2e;
                const float2 off = make_float2(-Ls, -Ls);
                const uint32_t ws[4] = {raw[u].x, raw[u].y, raw[u].z, raw[u].w};
                float2 pr[4];
#pragma unroll
                for (int j = 0; j < 4; ++j) {
                    const float2 x = fma2(make_float2(bf16_lo(ws[j]), bf16_hi(ws[j])), l2, off);
                    pr[j] = make_float2(ex2_fast(x.x), ex2_fast(x.y));
                }
                if (!full) {   // the last word of the row reaches into the padding
#pragma unroll
                    for (int j = 0; j < 4; ++j) {
                        if (col0 + 2 * j >= V) pr[j].x = 0.0f;
                        if (col0 + 2 * j + 1 >= V) pr[j].y = 0.0f;
                    }
                }
                const int64_t yy = static_cast<int64_t>(y) - yoff - col0;
                if (yy >= 0 && yy < VEC) {   // this word holds the label column
#pragma unroll
                    for (int j = 0; j < 4; ++j) {
                        if (yy == 2 * j) pr[j].x -= 1.0f;
                        if (yy == 2 * j + 1) pr[j].y -= 1.0f;
                    }
                }
#pragma unroll
                for (int j = 0; j < 4; ++j) cs[j] = add2(cs[j], pr[j]);
                *dst = make_uint4(cvt_bf16x2(pr[0].x, pr[0].y), cvt_bf16x2(pr[1].x, pr[1].y),
                                  cvt_bf16x2(pr[2].x, pr[2].y), cvt_bf16x2(pr[3].x, pr[3].y));
            }
        }
        float* out = colpart + static_cast<int64_t>(blockIdx.y) * V + col0;
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            if (col0 + 2 * j < V) out[2 * j] = cs[j].x;
            if (col0 + 2 * j + 1 < V) out[2 * j + 1] = cs[j].y;
        }
    } else {
        float csum[VEC];
#pragma unroll
        for (int k = 0; k < VEC; ++k) csum[k] = 0.0f;
        for (int64_t rb = r0; rb < r1; rb += UNROLL) {
            uint4 raw[UNROLL];
#pragma unroll
            for (int u = 0; u < UNROLL; ++u)
                if (rb + u < r1) raw[u] = *reinterpret_cast<const uint4*>(Z + (rb + u) * ldz + col0);
#pragma unroll
            for (int u = 0; u < UNROLL; ++u) {
                const int64_t r = rb + u;
                if (r >= r1) break;
                const int32_t y = labels[r];
                const bool valid = (y != ignore);
                const float L = lse[r];
                const uint32_t ws[4] = {raw[u].x, raw[u].y, raw[u].z, raw[u].w};
                float rv[VEC];
#pragma unroll
                for (int k = 0; k < VEC; ++k) {
                    const int64_t c = col0 + k;
                    float p = 0.0f;
                    if (valid && c < V) p = expf(__uint_as_float(ws[k]) - L);
                    if (valid && c + yoff == y) p -= 1.0f;
                    rv[k] = p;
                    csum[k] += p;
                }
                *reinterpret_cast<float4*>(Z + r * ldz + col0) = make_float4(rv[0], rv[1], rv[2], rv[3]);
            }
        }
#pragma unroll
        for (int k = 0; k < VEC; ++k)
            if (col0 + k < V) colpart[static_cast<int64_t>(blockIdx.y) * V + col0 + k] = csum[k];
    }
}

__global__ void __launch_bounds__(256) finish_sq_kernel(const float* __restrict__ colpart, int64_t nblocks, int64_t V,
                                                        float beta1, float* __restrict__ q,
                                                        float* __restrict__ s_out, float* __restrict__ qhat,
                                                        const DevScalars* sc) {
    pdl_enter();
    __shared__ float red[8][33];
    if (sc->status != 0) return;
    const int64_t j = static_cast<int64_t>(blockIdx.x) * 32 + (threadIdx.x & 31);
    const float acc = fixed_order_column_sum(colpart, nblocks, V, j, red);
    if (threadIdx.x >= 32 || j >= V) return;
    const float s = acc * sc->inv_nt;
    const float inv_bc1 = sc->inv_bc1;
    const float qn = beta1 * q[j] + (1.0f - beta1) * s;
    q[j] = qn;
    s_out[j] = s;
    qhat[j] = qn * inv_bc1;
}

__global__ void __launch_bounds__(1024) scalars_kernel(const float* __restrict__ ce, int64_t n,
                                                       const float* __restrict__ s_vec, int64_t V,
                                                       const float* __restrict__ rnorm, DevScalars* sc) {
    pdl_enter();
    __shared__ float red[32];
    if (sc->status != 0) return;
    float a = 0.0f;
    if (ce) {
        for (int64_t i = threadIdx.x; i < n; i += 1024) a += ce[i];
        a = block_sum<1024>(a, red);
    }
    float b = 0.0f;
    for (int64_t j = threadIdx.x; j < V; j += 1024) b += s_vec[j] * s_vec[j];
    b = block_sum<1024>(b, red);
    float c = 0.0f;
    if (rnorm) {
        for (int64_t i = threadIdx.x; i < n; i += 1024) c += rnorm[i];
        c = block_sum<1024>(c, red);
    }
    if (threadIdx.x == 0) {
        if (ce) sc->loss = a * sc->inv_nt;   // else set from the shards' summed CE
        sc->s_norm = sqrtf(b);
        sc->r_norm_mean = c * sc->inv_nt;
    }
}

// ||r_i|| of every row of R (0 on ignored rows, whose residual is zero): one
// warp per row, lane-strided fp32 sums reduced by a fixed shuffle tree.
template <typename T>
__global__ void __launch_bounds__(256) row_norm_kernel(const T* __restrict__ R, int64_t ldr, int64_t n, int64_t V,
                                                       float* __restrict__ rnorm, const DevScalars* sc) {
    pdl_enter();
    if (sc->status != 0) return;
    const int64_t row = (static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x) >> 5;
    const int l = threadIdx.x & 31;
    if (row >= n) return;
    const T* r = R + row * ldr;
    float a = 0.0f;
    for (int64_t j = l; j < V; j += 32) {
        const float x = ld_elem(r, j, sizeof(T) == 4);
        a = fmaf(x, x, a);
    }
    a = warp_sum(a);
    if (l == 0) rnorm[row] = sqrtf(a);
}

// Own-step moment and drift sums over a flat range (see bom_own_step_moment):
// per-thread fp32 sums, then per-block fp64 partials in a fixed slot each.
__global__ void __launch_bounds__(256) own_step_moment_kernel(float* __restrict__ M, const float* __restrict__ o,
                                                              const float* __restrict__ hv, float* __restrict__ mhat,
                                                              int64_t n, float beta1, float inv_bc1,
                                                              double* __restrict__ part) {
    pdl_enter();
    float s_dot = 0.0f, s_mm = 0.0f, s_hh = 0.0f, s_dd = 0.0f;
    auto one = [&](float& m, float oo, float h, float& mh) {
        m = fmaf(beta1, m, (1.0f - beta1) * oo);
        mh = m * inv_bc1;
        const float d = mh - h;
        s_dot = fmaf(mh, h, s_dot);
        s_mm = fmaf(mh, mh, s_mm);
        s_hh = fmaf(h, h, s_hh);
        s_dd = fmaf(d, d, s_dd);
    };
    // 16-byte words (all pointers are 16-byte aligned), two per thread in
    // flight (the words i and i + stride, in that order), then the tail
    const int64_t n4 = n >> 2;
    const int64_t stride = static_cast<int64_t>(gridDim.x) * blockDim.x;
    auto word = [&](int64_t i, float4 m, const float4& oo, const float4& h) {
        float4 mh;
        one(m.x, oo.x, h.x, mh.x);
        one(m.y, oo.y, h.y, mh.y);
        one(m.z, oo.z, h.z, mh.z);
        one(m.w, oo.w, h.w, mh.w);
        reinterpret_cast<float4*>(M)[i] = m;
        __stcs(reinterpret_cast<float4*>(mhat) + i, mh);
    };
    const float4 zero4 = make_float4(0.f, 0.f, 0.f, 0.f);
    int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x;
    for (; i + stride < n4; i += 2 * stride) {
        const int64_t j = i + stride;
        const float4 ma = reinterpret_cast<const float4*>(M)[i];
        const float4 mb = reinterpret_cast<const float4*>(M)[j];
        const float4 oa = __ldcs(reinterpret_cast<const float4*>(o) + i);
        const float4 ob = __ldcs(reinterpret_cast<const float4*>(o) + j);
        const float4 ha = hv ? __ldcs(reinterpret_cast<const float4*>(hv) + i) : zero4;
        const float4 hb = hv ? __ldcs(reinterpret_cast<const float4*>(hv) + j) : zero4;
        word(i, ma, oa, ha);
        word(j, mb, ob, hb);
    }
    if (i < n4)
        word(i, reinterpret_cast<const float4*>(M)[i], __ldcs(reinterpret_cast<const float4*>(o) + i),
             hv ? __ldcs(reinterpret_cast<const float4*>(hv) + i) : zero4);
    if (blockIdx.x == 0 && threadIdx.x < (n & 3)) {
        const int64_t i = (n4 << 2) + threadIdx.x;
        float m = M[i], mh;
        one(m, o[i], hv ? hv[i] : 0.0f, mh);
        M[i] = m;
        mhat[i] = mh;
    }
    if (!part) return;
    __shared__ double red[4][8];
    const int w = threadIdx.x >> 5, l = threadIdx.x & 31;
    const float v4[4] = {warp_sum(s_dot), warp_sum(s_mm), warp_sum(s_hh), warp_sum(s_dd)};
    if (l == 0)
        for (int k = 0; k < 4; ++k) red[k][w] = static_cast<double>(v4[k]);
    __syncthreads();
    if (threadIdx.x < 4) {
        double acc = 0.0;
        for (int k = 0; k < 8; ++k) acc += red[threadIdx.x][k];
        part[4 * static_cast<int64_t>(blockIdx.x) + threadIdx.x] = acc;
    }
}

// sums[k] += sum_b part[4b + k]: warp k, lane l adds blocks l, l + 32, ... in
// order, then a fixed shuffle tree (the order depends only on nblocks).
__global__ void drift_finish_kernel(const double* __restrict__ part, int nblocks, double* __restrict__ sums) {
    pdl_enter();
    const int k = threadIdx.x >> 5, l = threadIdx.x & 31;
    double acc = 0.0;
    for (int b = l; b < nblocks; b += 32) acc += part[4 * static_cast<int64_t>(b) + k];
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, o);
    if (l == 0) sums[k] += acc;
}

// part[b, j] = sum_{i in row range b} w_i X[i, j] (times Y[i, j] when Y is
// given, same layout as X); row range b is [b * rows_per, (b + 1) * rows_per).
// A block covers 32 x VEC columns of one row range: every warp reads 16-byte
// words of the same columns, the 8 warps take interleaved rows, and the 8 warp
// sums are added in a fixed order in shared memory (deterministic).  The host
// sizes the ranges so that the whole grid is one resident wave and each block
// streams many rows (colsum_rows_per).
template <typename T>
__device__ __forceinline__ float word_elem(const uint4& w, int k) {
    const uint32_t v = (k >> (sizeof(T) == 2 ? 1 : 0)) == 0   ? w.x
                       : (k >> (sizeof(T) == 2 ? 1 : 0)) == 1 ? w.y
                       : (k >> (sizeof(T) == 2 ? 1 : 0)) == 2 ? w.z
                                                              : w.w;
    if constexpr (sizeof(T) == 2)
        return __uint_as_float((k & 1) ? (v & 0xFFFF0000u) : (v << 16));
    else
        return __uint_as_float(v);
}

// With `out` given (a single row range), the block writes the final column
// sums, scaled and in out's dtype, instead of partials.
template <typename T, bool HAS_Y>
__global__ void __launch_bounds__(256, 3) colsum_part_kernel(const T* __restrict__ X, const T* __restrict__ Y,
                                                             int64_t ldx, int64_t n, int64_t rows_per,
                                                             int64_t d, const int32_t* __restrict__ labels,
                                                             int32_t ignore, const float* __restrict__ wvec,
                                                             float* __restrict__ part, void* __restrict__ out,
                                                             int out_f32, float scale, const DevScalars* sc) {
    pdl_enter();
    constexpr int VEC = 16 / sizeof(T);
    // rows in flight per warp step: 8 words per thread (4 of X and 4 of Y)
    constexpr int U = HAS_Y ? 4 : 8;
    __shared__ float red[8][32 * VEC];
    if (sc->status != 0) return;
    const int w = threadIdx.x >> 5, l = threadIdx.x & 31;
    const int64_t c0 = static_cast<int64_t>(blockIdx.x) * (32 * VEC) + l * VEC;
    const int64_t r0 = static_cast<int64_t>(blockIdx.y) * rows_per;
    const int64_t r1 = min(r0 + rows_per, n);
    float acc[VEC];
#pragma unroll
    for (int k = 0; k < VEC; ++k) acc[k] = 0.0f;
    auto weight = [&](int64_t r) {
        if (labels) return labels[r] != ignore ? 1.0f : 0.0f;
        return wvec ? wvec[r] : 1.0f;
    };
    if (c0 + VEC <= d && (ldx % VEC) == 0) {
        const T* px = X + c0;
        const T* py = HAS_Y ? Y + c0 : nullptr;
        int64_t r = r0 + w;
        for (; r + 8 * (U - 1) < r1; r += 8 * U) {
            uint4 a[U], b[HAS_Y ? U : 1];
            float wt[U];
#pragma unroll
            for (int u = 0; u < U; ++u) {
                const int64_t off = (r + 8 * u) * ldx;
                a[u] = __ldcs(reinterpret_cast<const uint4*>(px + off));
                if constexpr (HAS_Y) b[u] = __ldcs(reinterpret_cast<const uint4*>(py + off));
                wt[u] = weight(r + 8 * u);
            }
#pragma unroll
            for (int u = 0; u < U; ++u) {
#pragma unroll
                for (int k = 0; k < VEC; ++k) {
                    float x = word_elem<T>(a[u], k);
                    if constexpr (HAS_Y) x *= word_elem<T>(b[u], k);
                    acc[k] = fmaf(wt[u], x, acc[k]);
                }
            }
        }
        for (; r < r1; r += 8) {
            const int64_t off = r * ldx;
            const uint4 a = __ldcs(reinterpret_cast<const uint4*>(px + off));
            uint4 b = a;
            if constexpr (HAS_Y) b = __ldcs(reinterpret_cast<const uint4*>(py + off));
            const float wr = weight(r);
#pragma unroll
            for (int k = 0; k < VEC; ++k) {
                float x = word_elem<T>(a, k);
                if constexpr (HAS_Y) x *= word_elem<T>(b, k);
                acc[k] = fmaf(wr, x, acc[k]);
            }
        }
    } else if (c0 < d) {
        // ragged last column group or a pitch that breaks 16-byte alignment
        for (int64_t r = r0 + w; r < r1; r += 8) {
            const float wr = weight(r);
#pragma unroll
            for (int k = 0; k < VEC; ++k) {
                if (c0 + k >= d) break;
                float x = static_cast<float>(X[r * ldx + c0 + k]);
                if constexpr (HAS_Y) x *= static_cast<float>(Y[r * ldx + c0 + k]);
                acc[k] = fmaf(wr, x, acc[k]);
            }
        }
    }
#pragma unroll
    for (int k = 0; k < VEC; ++k) red[w][l * VEC + k] = acc[k];
    __syncthreads();
    for (int j = threadIdx.x; j < 32 * VEC; j += 256) {
        const int64_t c = static_cast<int64_t>(blockIdx.x) * (32 * VEC) + j;
        if (c >= d) continue;
        float a = 0.0f;
#pragma unroll
        for (int k = 0; k < 8; ++k) a += red[k][j];
        if (out != nullptr)
            st_elem(out, c, out_f32, a * scale);
        else
            part[static_cast<int64_t>(blockIdx.y) * d + c] = a;
    }
}

__global__ void __launch_bounds__(256) colsum_finish_kernel(const float* __restrict__ part, int64_t nblocks,
                                                            int64_t d, float scale, void* __restrict__ out,
                                                            int out_f32, const DevScalars* sc) {
    pdl_enter();
    __shared__ float red[8][33];
    if (sc->status != 0) return;
    const int64_t j = static_cast<int64_t>(blockIdx.x) * 32 + (threadIdx.x & 31);
    const float a = fixed_order_column_sum(part, nblocks, d, j, red);
    if (threadIdx.x < 32 && j < d) st_elem(out, j, out_f32, a * scale);
}

__global__ void axpby_kernel(const float* __restrict__ s, const float* __restrict__ qh, float a, float b, int64_t V,
                             void* __restrict__ out, int out_f32, const DevScalars* sc) {
    pdl_enter();
    if (sc->status != 0) return;
    const int64_t j = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x;
    if (j >= V) return;
    st_elem(out, j, out_f32, a * s[j] + b * qh[j]);
}

// ---------------------------------------------------------------------------
// Row-sharded step (Algorithm 1's batch mean over I_t split by rows).  A shard
// writes the sums that couple its rows to the others: the column sums of its
// residuals, its CE sum, its |I_t^shard| and an error flag, in fp64 so that
// any number of shards adds them exactly enough (the counts exactly).
// xch[j] for j < V: sum_{i in I_t^shard} r_ij (the fixed-order fp32 column sum
// of the residual pass's partials); nothing is read when the shard latched an
// error (zeros are written).
__global__ void __launch_bounds__(256) shard_colsum_kernel(const float* __restrict__ colpart, int64_t nblocks,
                                                           int64_t V, double* __restrict__ xch,
                                                           const DevScalars* sc) {
    pdl_enter();
    __shared__ float red[8][33];
    const bool ok = sc->status == 0;
    const int64_t j = static_cast<int64_t>(blockIdx.x) * 32 + (threadIdx.x & 31);
    const float acc = fixed_order_column_sum(colpart, ok ? nblocks : 0, V, j, red);
    if (threadIdx.x < 32 && j < V) xch[j] = ok ? static_cast<double>(acc) : 0.0;
}

// xch[V] = sum_{i in I_t^shard} CE_i (fixed order), xch[V+1] = |I_t^shard|,
// xch[V+2] = 1 when this shard latched an error, else 0.
__global__ void __launch_bounds__(1024) shard_scalars_out_kernel(const float* __restrict__ ce, int64_t n,
                                                                 int64_t V, double* __restrict__ xch,
                                                                 const DevScalars* sc) {
    pdl_enter();
    __shared__ float red[32];
    const bool ok = sc->status == 0;
    float a = 0.0f;
    if (ok)
        for (int64_t i = threadIdx.x; i < n; i += 1024) a += ce[i];
    a = block_sum<1024>(a, red);
    if (threadIdx.x == 0) {
        xch[V] = ok ? static_cast<double>(a) : 0.0;
        xch[V + 1] = ok ? static_cast<double>(sc->n_t) : 0.0;
        xch[V + 2] = ok ? 0.0 : 1.0;
    }
}

// The second half of a sharded step begins here, from the summed vector:
// N_t of the whole batch, the cotangent coefficients, the loss, the step
// scalars and this shard's share N_t^shard / N_t.  Any shard's error stops
// every shard (BOM_ESHARD where this one had none), and so does N_t = 0.
__global__ void shard_scalars_in_kernel(const double* __restrict__ xch, int64_t V, float lambda,
                                        const StepScalarsIn st, DevScalars* sc) {
    pdl_enter();
    if (threadIdx.x != 0) return;
    const int32_t n_loc = sc->n_t;
    const double nt_d = xch[V + 1];
    const int64_t nt = nt_d >= 0.0 && nt_d < 4.0e18 ? static_cast<int64_t>(nt_d) : -1;
    if (xch[V + 2] != 0.0)
        latch_status(sc, BOM_ESHARD);
    else if (nt == 0)
        latch_status(sc, BOM_EEMPTY);
    else if (nt < 0 || nt > INT32_MAX || static_cast<double>(nt) != nt_d)
        latch_status(sc, BOM_EINVAL);   // not a sum of row counts
    const bool ok = sc->status == 0;
    sc->n_t = ok ? static_cast<int32_t>(nt) : 0;
    const float inv = ok ? 1.0f / static_cast<float>(nt) : 0.0f;
    sc->inv_nt = inv;
    sc->shard_frac = ok ? static_cast<float>(static_cast<double>(n_loc) / nt_d) : 0.0f;
    sc->coef_r[0] = (1.0f - lambda) * inv;
    sc->coef_q[0] = lambda * inv;
    sc->coef_r[1] = inv;
    sc->coef_q[1] = 0.0f;
    sc->coef_r[2] = 0.0f;
    sc->coef_q[2] = inv;
    sc->coef_r[3] = 0.0f;
    sc->coef_q[3] = inv;
    float bc1 = st.inv_bc1, bc2 = st.inv_bc2;
    if (st.t_dev != nullptr) {
        const int64_t t = *st.t_dev;
        if (t < 1) {
            latch_status(sc, BOM_EINVAL);
        } else {
            bc1 = inv_bias_correction(st.beta1, t);
            bc2 = inv_bias_correction(st.beta2, t);
        }
    }
    sc->lr = st.lr_dev != nullptr ? *st.lr_dev : st.lr;
    sc->inv_bc1 = bc1;
    sc->inv_bc2 = bc2;
    sc->loss = ok ? static_cast<float>(xch[V] / nt_d) : 0.0f;
    sc->s_norm = 0.0f;
    sc->r_norm_mean = 0.0f;
}

// s_j = N_t^-1 xch[j], q_j <- beta1 q_j + (1-beta1) s_j, qhat_j = q_j / (1-beta1^t)
// from the summed vector (every shard forms the same q), and this shard's
// share s^shard_j = N_t^-1 sum_{i in I_t^shard} r_ij from its own partials.
__global__ void __launch_bounds__(256) shard_finish_sq_kernel(const double* __restrict__ xch,
                                                              const float* __restrict__ colpart, int64_t nblocks,
                                                              int64_t V, float beta1, float* __restrict__ q,
                                                              float* __restrict__ s_out, float* __restrict__ qhat,
                                                              float* __restrict__ s_shard, const DevScalars* sc) {
    pdl_enter();
    __shared__ float red[8][33];
    if (sc->status != 0) return;
    const int64_t j = static_cast<int64_t>(blockIdx.x) * 32 + (threadIdx.x & 31);
    const float loc = fixed_order_column_sum(colpart, nblocks, V, j, red);
    if (threadIdx.x >= 32 || j >= V) return;
    const float inv = sc->inv_nt;
    const float s = static_cast<float>(xch[j]) * inv;
    const float qn = beta1 * q[j] + (1.0f - beta1) * s;
    q[j] = qn;
    s_out[j] = s;
    qhat[j] = qn * sc->inv_bc1;
    s_shard[j] = loc * inv;
}

// This shard's share of the head bias numerator: a s^shard + b (N_t^shard / N_t) qhat.
__global__ void shard_bias_kernel(const float* __restrict__ s_shard, const float* __restrict__ qh, float a, float b,
                                  int64_t V, void* __restrict__ out, int out_f32, const DevScalars* sc) {
    pdl_enter();
    if (sc->status != 0) return;
    const int64_t j = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x;
    if (j >= V) return;
    st_elem(out, j, out_f32, a * s_shard[j] + b * sc->shard_frac * qh[j]);
}

// ---------------------------------------------------------------------------
// Vocabulary-sharded step: the head's output columns split over shards.  The
// residual r_ij = exp(z_ij - lse_i) - [j = y_i] (Algorithm 1) couples a row's
// columns only through its log-sum-exp, so each shard sends one number per
// row, and s_t, q_t and qhat_t of its columns need no exchange at all.
//
// This shard's part of each row's log-sum-exp, log sum_{j in shard} exp(z_ij),
// from the per-tile (max, sum exp) pairs of the logits epilogue (one warp per
// row, the pairs in tile order).  A shard that latched an error writes NaN on
// every row, and a row whose part is not finite latches BOM_ENONFINITE and
// writes NaN: the shards that combine the parts stop on it.
__global__ void __launch_bounds__(256) vshard_lse_part_kernel(const float2* __restrict__ stats, int64_t ntiles,
                                                              int64_t n, float* __restrict__ lse_part,
                                                              DevScalars* sc) {
    pdl_enter();
    const int64_t row = (static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x) >> 5;
    const int l = threadIdx.x & 31;
    if (row >= n) return;
    if (sc->status != 0) {
        if (l == 0) lse_part[row] = __int_as_float(0x7fc00000);
        return;
    }
    const float2* st = stats + row * ntiles;
    float m = -INFINITY;
    for (int64_t t = l; t < ntiles; t += 32) m = fmaxf(m, st[t].x);
    m = warp_max(m);
    float s = 0.0f;
    for (int64_t t = l; t < ntiles; t += 32) {
        const float2 p = st[t];
        if (p.x != -INFINITY) s += p.y * expf(p.x - m);
    }
    s = warp_sum(s);
    if (l == 0) {
        const float L = m + logf(s);
        if (!isfinite(L)) latch_status(sc, BOM_ENONFINITE);
        lse_part[row] = isfinite(L) ? L : __int_as_float(0x7fc00000);
    }
}

// Row log-sum-exp from every shard's part, combined in shard order (every
// shard computes the same float): lse_i = M + log sum_r exp(part[r, i] - M),
// M = max_r part[r, i].  ce_i = lse_i - z_{i,y_i} on the supervised rows whose
// label column this shard holds (y_i - v0 in [0, Vloc)), 0 on the others, so
// the shards' CE sums add up to the batch's.  A NaN part (a shard that
// stopped) latches BOM_ESHARD.  Thread 0 also writes the step scalars (host t,
// or the device step counter), which the first half had no t for.
__global__ void __launch_bounds__(256) vshard_lse_kernel(const float* __restrict__ parts, int32_t nsh, int64_t n,
                                                         const void* __restrict__ Z, int z_f32, int64_t ldz,
                                                         int64_t v0, int64_t Vloc,
                                                         const int32_t* __restrict__ labels, int32_t ignore,
                                                         float* __restrict__ lse, float* __restrict__ ce,
                                                         const StepScalarsIn st, DevScalars* sc) {
    pdl_enter();
    if (blockIdx.x == 0 && threadIdx.x == 0) {
        float bc1 = st.inv_bc1;
        if (st.t_dev != nullptr) {
            const int64_t t = *st.t_dev;
            if (t < 1)
                latch_status(sc, BOM_EINVAL);
            else
                bc1 = inv_bias_correction(st.beta1, t);
        }
        sc->inv_bc1 = bc1;
    }
    if (sc->status != 0) return;
    const int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x;
    if (i >= n) return;
    float M = -INFINITY;
    bool stopped = false;
    for (int r = 0; r < nsh; ++r) {
        const float p = parts[static_cast<int64_t>(r) * n + i];
        stopped = stopped || isnan(p);
        M = fmaxf(M, p);
    }
    if (stopped) {
        latch_status(sc, BOM_ESHARD);
        return;
    }
    float S = 0.0f;
    for (int r = 0; r < nsh; ++r) S += expf(parts[static_cast<int64_t>(r) * n + i] - M);
    const float L = M + logf(S);
    const int32_t y = labels[i];
    const int64_t yl = static_cast<int64_t>(y) - v0;
    const bool owned = y != ignore && yl >= 0 && yl < Vloc;
    const float zy = owned ? ld_elem(Z, i * ldz + yl, z_f32) : 0.0f;
    lse[i] = L;
    ce[i] = owned ? L - zy : 0.0f;
    if (!isfinite(L) || (owned && !isfinite(zy))) latch_status(sc, BOM_ENONFINITE);
}

// dst = src over n elements (fp32 to bf16 by round to nearest even, or an
// fp32 copy): the summed input cotangent of the head, in the compute dtype the
// backbone's backward reads.  Four elements per thread from 16-byte aligned
// buffers, the last n mod 4 one by one.
__global__ void __launch_bounds__(256) cast_f32_kernel(const float* __restrict__ src, void* __restrict__ dst,
                                                       int64_t n, int dst_f32, const DevScalars* sc) {
    pdl_enter();
    if (sc->status != 0) return;
    const int64_t n4 = n / 4;
    const int64_t stride = static_cast<int64_t>(gridDim.x) * blockDim.x;
    const int64_t k0 = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x;
    for (int64_t k = k0; k < n4; k += stride) {
        const float4 v = reinterpret_cast<const float4*>(src)[k];
        if (dst_f32)
            reinterpret_cast<float4*>(dst)[k] = v;
        else
            reinterpret_cast<uint2*>(dst)[k] = make_uint2(cvt_bf16x2(v.x, v.y), cvt_bf16x2(v.z, v.w));
    }
    for (int64_t k = 4 * n4 + k0; k < n; k += stride) st_elem(dst, k, dst_f32, src[k]);
}

inline unsigned cdiv(int64_t a, int64_t b) { return static_cast<unsigned>((a + b - 1) / b); }

}  // namespace

void launch_labels_scan(const int32_t* labels, int64_t n, int64_t V, int32_t ignore, float lambda,
                        const StepScalarsIn& st, DevScalars* sc, cudaStream_t s, bool allow_empty) {
    launch_k(labels_scan_kernel, dim3(1), dim3(1024), 0, s, labels, n, V, ignore, lambda, st, allow_empty ? 1 : 0, sc);
    count_launch();
}

void launch_advance_step(int64_t* t_dev, const DevScalars* sc, cudaStream_t s) {
    launch_k(advance_step_kernel, dim3(1), dim3(32), 0, s, t_dev, sc); count_launch();
}

void launch_row_stats_f32(const float* Z, int64_t ldz, int64_t n, int64_t V, float* stats, const DevScalars* sc,
                          cudaStream_t s) {
    launch_k(row_stats_f32_kernel, dim3(cdiv(n * 32, 256)), dim3(256), 0, s, Z, ldz, n, V, reinterpret_cast<float2*>(stats), sc); count_launch();
}

void launch_row_lse(const void* Z, int z_f32, int64_t ldz, int64_t n, int64_t V, const float* stats, int64_t ntiles,
                    const int32_t* labels, int32_t ignore, float* lse, float* ce, DevScalars* sc,
                    cudaStream_t s) {
    launch_k(row_lse_kernel, dim3(cdiv(n * 32, 256)), dim3(256), 0, s, Z, z_f32, ldz, n, V, reinterpret_cast<const float2*>(stats),
                                                      ntiles, labels, ignore, lse, ce, sc); count_launch();
}

void launch_residual(void* Z, int z_f32, int64_t ldz, int64_t n, int64_t V, const float* lse, const int32_t* labels,
                     int32_t ignore, float* colpart, const DevScalars* sc, cudaStream_t s, int64_t yoff) {
    if (z_f32) {
        dim3 grid(cdiv(ldz, 256 * 4), static_cast<unsigned>(resid_blocks(n)));
        launch_k(residual_kernel<float, 4>, dim3(grid), dim3(256), 0, s, static_cast<float*>(Z), ldz, n, V, lse, labels, ignore,
                                                       yoff, colpart, sc); count_launch();
    } else {
        dim3 grid(cdiv(ldz, 256 * 8), static_cast<unsigned>(resid_blocks(n)));
        launch_k(residual_kernel<__nv_bfloat16, 8>, dim3(grid), dim3(256), 0, s, static_cast<__nv_bfloat16*>(Z), ldz, n, V, lse,
                                                               labels, ignore, yoff, colpart, sc); count_launch();
    }
}

void launch_finish_sq(const float* colpart, int64_t nblocks, int64_t V, float beta1, float* q,
                      float* s_out, float* qhat, DevScalars* sc, cudaStream_t s) {
    launch_k(finish_sq_kernel, dim3(cdiv(V, 32)), dim3(256), 0, s, colpart, nblocks, V, beta1, q, s_out, qhat, sc); count_launch();
}

void launch_scalars(const float* ce, int64_t n, const float* s_vec, int64_t V, const float* rnorm, DevScalars* sc,
                    cudaStream_t s) {
    launch_k(scalars_kernel, dim3(1), dim3(1024), 0, s, ce, n, s_vec, V, rnorm, sc); count_launch();
}

void launch_row_norm(const void* R, int r_f32, int64_t ldr, int64_t n, int64_t V, float* rnorm, const DevScalars* sc,
                     cudaStream_t s) {
    const unsigned grid = static_cast<unsigned>(cdiv(n * 32, 256));
    if (r_f32)
        launch_k(row_norm_kernel<float>, dim3(grid), dim3(256), 0, s, static_cast<const float*>(R), ldr, n, V, rnorm, sc);
    else
        launch_k(row_norm_kernel<__nv_bfloat16>, dim3(grid), dim3(256), 0, s, static_cast<const __nv_bfloat16*>(R), ldr, n, V, rnorm,
                                                             sc);
    count_launch();
}

int own_step_blocks(int64_t n, int sms) {
    int64_t b = cdiv(n, 256 * 16);
    const int64_t cap = std::min<int64_t>(4 * static_cast<int64_t>(sms > 0 ? sms : 1), kOwnStepMaxBlocks);
    b = b < cap ? b : cap;
    return static_cast<int>(b < 1 ? 1 : b);
}

void launch_own_step_moment(float* M, const float* o, const float* hv, float* mhat, int64_t n, float beta1,
                            float inv_bc1, double* part, int nblocks, double* sums, cudaStream_t s) {
    launch_k(own_step_moment_kernel, dim3(nblocks), dim3(256), 0, s, M, o, hv, mhat, n, beta1, inv_bc1, sums ? part : nullptr);
    count_launch();
    if (sums) {
        launch_k(drift_finish_kernel, dim3(1), dim3(128), 0, s, part, nblocks, sums);
        count_launch();
    }
}

// Rows per block of the column reduction: the fewest row ranges that still
// give every SM three blocks (one resident wave), and never more ranges than
// row_blocks(n), which is what callers size the partial buffer for.  Whole
// multiples of 64 rows keep the 8 warps' 8-row unrolled steps full.
static int64_t colsum_rows_per(int64_t n, int64_t col_groups, int sms) {
    const int64_t want = std::max<int64_t>(1, (3 * static_cast<int64_t>(sms > 0 ? sms : 1)) / std::max<int64_t>(col_groups, 1));
    const int64_t ranges = std::min<int64_t>(row_blocks(n), want);
    int64_t per = (n + ranges - 1) / ranges;
    per = (per + 63) / 64 * 64;
    return std::max<int64_t>(per, kRowBlock);
}

void launch_colsum(const void* X, int x_f32, int64_t ldx, int64_t n, int64_t d, const int32_t* labels,
                   int32_t ignore, const float* wvec, float scale, float* part, void* out, int out_f32,
                   const DevScalars* sc, cudaStream_t s) {
    launch_colsum2(X, nullptr, x_f32, ldx, n, d, labels, ignore, wvec, scale, part, out, out_f32, sc, s);
}

void launch_colsum2(const void* X, const void* Y, int x_f32, int64_t ldx, int64_t n, int64_t d,
                    const int32_t* labels, int32_t ignore, const float* wvec, float scale, float* part, void* out,
                    int out_f32, const DevScalars* sc, cudaStream_t s) {
    const int64_t cols_per_block = x_f32 ? 128 : 256;
    // a batch within one row range: its blocks write the result directly and
    // the finishing launch is skipped
    const bool single = n <= kRowBlock;
    const int64_t rows_per = single ? (n > 0 ? n : 1) : colsum_rows_per(n, cdiv(d, cols_per_block), device_sm_count());
    const int64_t nb = (n + rows_per - 1) / rows_per;
    void* const direct = single ? out : nullptr;
    dim3 grid(cdiv(d, cols_per_block), static_cast<unsigned>(nb > 0 ? nb : 1));
    if (x_f32) {
        auto x = static_cast<const float*>(X);
        auto y = static_cast<const float*>(Y);
        if (Y)
            launch_k(colsum_part_kernel<float, true>, dim3(grid), dim3(256), 0, s, x, y, ldx, n, rows_per, d, labels,
                     ignore, wvec, part, direct, out_f32, scale, sc);
        else
            launch_k(colsum_part_kernel<float, false>, dim3(grid), dim3(256), 0, s, x, y, ldx, n, rows_per, d, labels,
                     ignore, wvec, part, direct, out_f32, scale, sc);
    } else {
        auto x = static_cast<const __nv_bfloat16*>(X);
        auto y = static_cast<const __nv_bfloat16*>(Y);
        if (Y)
            launch_k(colsum_part_kernel<__nv_bfloat16, true>, dim3(grid), dim3(256), 0, s, x, y, ldx, n, rows_per, d,
                     labels, ignore, wvec, part, direct, out_f32, scale, sc);
        else
            launch_k(colsum_part_kernel<__nv_bfloat16, false>, dim3(grid), dim3(256), 0, s, x, y, ldx, n, rows_per,
                     d, labels, ignore, wvec, part, direct, out_f32, scale, sc);
    }
    count_launch();
    if (single) return;
    launch_k(colsum_finish_kernel, dim3(cdiv(d, 32)), dim3(256), 0, s, part, nb, d, scale, out, out_f32, sc);
    count_launch();
}

void launch_axpby(const float* s_vec, const float* qhat, float a, float b, int64_t V, void* out, int out_f32,
                  const DevScalars* sc, cudaStream_t s) {
    launch_k(axpby_kernel, dim3(cdiv(V, 256)), dim3(256), 0, s, s_vec, qhat, a, b, V, out, out_f32, sc); count_launch();
}

void launch_shard_sums(const float* colpart, int64_t nblocks, const float* ce, int64_t n, int64_t V, double* xch,
                       const DevScalars* sc, cudaStream_t s) {
    launch_k(shard_colsum_kernel, dim3(cdiv(V, 32)), dim3(256), 0, s, colpart, nblocks, V, xch, sc);
    count_launch();
    launch_k(shard_scalars_out_kernel, dim3(1), dim3(1024), 0, s, ce, n, V, xch, sc);
    count_launch();
}

void launch_shard_scalars_in(const double* xch, int64_t V, float lambda, const StepScalarsIn& st, DevScalars* sc,
                             cudaStream_t s) {
    launch_k(shard_scalars_in_kernel, dim3(1), dim3(32), 0, s, xch, V, lambda, st, sc);
    count_launch();
}

void launch_shard_finish_sq(const double* xch, const float* colpart, int64_t nblocks, int64_t V, float beta1,
                            float* q, float* s_out, float* qhat, float* s_shard, const DevScalars* sc,
                            cudaStream_t s) {
    launch_k(shard_finish_sq_kernel, dim3(cdiv(V, 32)), dim3(256), 0, s, xch, colpart, nblocks, V, beta1, q, s_out,
             qhat, s_shard, sc);
    count_launch();
}

void launch_shard_bias(const float* s_shard, const float* qhat, float a, float b, int64_t V, void* out, int out_f32,
                       const DevScalars* sc, cudaStream_t s) {
    launch_k(shard_bias_kernel, dim3(cdiv(V, 256)), dim3(256), 0, s, s_shard, qhat, a, b, V, out, out_f32, sc);
    count_launch();
}

void launch_vshard_lse_part(const float* stats, int64_t ntiles, int64_t n, float* lse_part, DevScalars* sc,
                            cudaStream_t s) {
    launch_k(vshard_lse_part_kernel, dim3(cdiv(n * 32, 256)), dim3(256), 0, s, reinterpret_cast<const float2*>(stats),
             ntiles, n, lse_part, sc);
    count_launch();
}

void launch_vshard_lse(const float* parts, int32_t nsh, int64_t n, const void* Z, int z_f32, int64_t ldz, int64_t v0,
                       int64_t Vloc, const int32_t* labels, int32_t ignore, float* lse, float* ce,
                       const StepScalarsIn& st, DevScalars* sc, cudaStream_t s) {
    launch_k(vshard_lse_kernel, dim3(cdiv(n, 256)), dim3(256), 0, s, parts, nsh, n, Z, z_f32, ldz, v0, Vloc, labels,
             ignore, lse, ce, st, sc);
    count_launch();
}

void launch_cast_f32(const float* src, void* dst, int64_t n, int dst_f32, const DevScalars* sc, cudaStream_t s) {
    const int64_t n4 = n / 4;
    int64_t blocks = cdiv(n4 > 0 ? n4 : 1, 256);
    if (blocks > 8 * device_sm_count()) blocks = 8 * device_sm_count();
    launch_k(cast_f32_kernel, dim3(static_cast<unsigned>(blocks)), dim3(256), 0, s, src, dst, n, dst_f32, sc);
    count_launch();
}

}  // namespace bom
