// Task-space part of the BOM step (Algorithm 1, residual / EMA steps):
// label scan and N_t, row log-sum-exp from the logits epilogue's per-tile
// statistics, the residual pass r = softmax(z) - onehot(y) with deterministic
// column partial sums, s_t and the q_t EMA with bias correction, and the
// column reductions colsum_{I_t}(H), W^T qhat and bias gradients.
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
    float a0 = 0.0f, a1 = 0.0f, a2 = 0.0f, a3 = 0.0f;
    if (col < ncols) {
        int64_t b = w;
        for (; b + 24 < nblocks; b += 32) {
            a0 += part[b * ncols + col];
            a1 += part[(b + 8) * ncols + col];
            a2 += part[(b + 16) * ncols + col];
            a3 += part[(b + 24) * ncols + col];
        }
        for (; b < nblocks; b += 8) a0 += part[b * ncols + col];
    }
    red[w][l] = (a0 + a1) + (a2 + a3);
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

__global__ void labels_scan_kernel(const int32_t* __restrict__ labels, int64_t n, int64_t V, int32_t ignore,
                                   float lambda, DevScalars* sc) {
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
        else if (c == 0)
            latch_status(sc, BOM_EEMPTY);
        const float inv = c > 0 ? 1.0f / static_cast<float>(c) : 0.0f;
        sc->inv_nt = inv;
        sc->coef_r[0] = (1.0f - lambda) * inv;  // u pass: N_t^-1 (1-lambda) r_i
        sc->coef_q[0] = lambda * inv;           //         N_t^-1 lambda qhat
        sc->coef_r[1] = inv;                    // g pass: N_t^-1 r_i
        sc->coef_q[1] = 0.0f;
        sc->coef_r[2] = 0.0f;                   // h pass: N_t^-1 qhat
        sc->coef_q[2] = inv;
        sc->loss = 0.0f;
        sc->s_norm = 0.0f;
    }
}

// One warp per row.
__global__ void row_stats_f32_kernel(const float* __restrict__ Z, int64_t ldz, int64_t n, int64_t V,
                                     float2* __restrict__ stats, const DevScalars* sc) {
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
                               int32_t ignore, float* __restrict__ lse, float* __restrict__ ce, const DevScalars* sc) {
    if (sc->status != 0) return;
    const int64_t row = (static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x) >> 5;
    const int l = threadIdx.x & 31;
    if (row >= n) return;
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
        lse[row] = L;
        const int32_t y = labels[row];
        float c = 0.0f;
        if (y != ignore && y >= 0 && y < V) c = L - ld_elem(Z, row * ldz + y, z_f32);
        ce[row] = c;
    }
}

// Block: 256 threads x VEC consecutive columns (one 16-byte word each) of
// kResidRows rows.  The words of UNROLL rows are loaded before any is used and
// stay packed until then, so a thread keeps 128 bytes in flight with few
// registers and three blocks fit on an SM.
template <typename T, int VEC>
__global__ void __launch_bounds__(256, 3) residual_kernel(T* __restrict__ Z, int64_t ldz, int64_t n, int64_t V,
                                                          const float* __restrict__ lse,
                                                          const int32_t* __restrict__ labels, int32_t ignore,
                                                          float* __restrict__ colpart, const DevScalars* sc) {
    if (sc->status != 0) return;
    const int64_t col0 = (static_cast<int64_t>(blockIdx.x) * 256 + threadIdx.x) * VEC;
    const int64_t r0 = static_cast<int64_t>(blockIdx.y) * kResidRows;
    const int64_t r1 = min(r0 + kResidRows, n);
    float csum[VEC];
#pragma unroll
    for (int k = 0; k < VEC; ++k) csum[k] = 0.0f;
    if (col0 < ldz) {
        constexpr int UNROLL = 8;
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
                // bf16 logits: exp2 of a pre-scaled argument (the result is
                // stored in bf16); fp32 logits keep the accurate expf.
                const float Ls = L * 1.4426950408889634f;
                const uint32_t ws[4] = {raw[u].x, raw[u].y, raw[u].z, raw[u].w};
                float z[VEC];
                if constexpr (sizeof(T) == 2) {
#pragma unroll
                    for (int j = 0; j < 4; ++j) {
                        z[2 * j] = __uint_as_float(ws[j] << 16);
                        z[2 * j + 1] = __uint_as_float(ws[j] & 0xFFFF0000u);
                    }
                } else {
#pragma unroll
                    for (int j = 0; j < 4; ++j) z[j] = __uint_as_float(ws[j]);
                }
                float rv[VEC];
#pragma unroll
                for (int k = 0; k < VEC; ++k) {
                    const int64_t c = col0 + k;
                    float p = 0.0f;
                    if (valid && c < V)
                        p = (sizeof(T) == 2) ? exp2f(fmaf(z[k], 1.4426950408889634f, -Ls)) : expf(z[k] - L);
                    if (valid && c == y) p -= 1.0f;
                    rv[k] = p;
                    csum[k] += p;
                }
                T* dst = Z + r * ldz + col0;
                if constexpr (sizeof(T) == 2) {
                    *reinterpret_cast<uint4*>(dst) = make_uint4(pack_bf16x2(rv[0], rv[1]), pack_bf16x2(rv[2], rv[3]),
                                                                pack_bf16x2(rv[4], rv[5]), pack_bf16x2(rv[6], rv[7]));
                } else {
                    *reinterpret_cast<float4*>(dst) = make_float4(rv[0], rv[1], rv[2], rv[3]);
                }
            }
        }
#pragma unroll
        for (int k = 0; k < VEC; ++k)
            if (col0 + k < V) colpart[static_cast<int64_t>(blockIdx.y) * V + col0 + k] = csum[k];
    }
}

__global__ void __launch_bounds__(256) finish_sq_kernel(const float* __restrict__ colpart, int64_t nblocks, int64_t V,
                                                        float beta1, float inv_bc1, float* __restrict__ q,
                                                        float* __restrict__ s_out, float* __restrict__ qhat,
                                                        const DevScalars* sc) {
    __shared__ float red[8][33];
    if (sc->status != 0) return;
    const int64_t j = static_cast<int64_t>(blockIdx.x) * 32 + (threadIdx.x & 31);
    const float acc = fixed_order_column_sum(colpart, nblocks, V, j, red);
    if (threadIdx.x >= 32 || j >= V) return;
    const float s = acc * sc->inv_nt;
    const float qn = beta1 * q[j] + (1.0f - beta1) * s;
    q[j] = qn;
    s_out[j] = s;
    qhat[j] = qn * inv_bc1;
}

__global__ void __launch_bounds__(1024) scalars_kernel(const float* __restrict__ ce, int64_t n,
                                                       const float* __restrict__ s_vec, int64_t V, DevScalars* sc) {
    __shared__ float red[32];
    if (sc->status != 0) return;
    float a = 0.0f;
    for (int64_t i = threadIdx.x; i < n; i += 1024) a += ce[i];
    a = block_sum<1024>(a, red);
    float b = 0.0f;
    for (int64_t j = threadIdx.x; j < V; j += 1024) b += s_vec[j] * s_vec[j];
    b = block_sum<1024>(b, red);
    if (threadIdx.x == 0) {
        sc->loss = a * sc->inv_nt;
        sc->s_norm = sqrtf(b);
    }
}

// part[b, j] = sum_{i in row block b} w_i X[i, j].  A block covers 32 x VEC
// columns of one row block: every warp reads 16-byte words of the same
// columns, the 8 warps take interleaved rows, and the 8 warp sums are added
// in a fixed order in shared memory (deterministic).
template <typename T>
__global__ void __launch_bounds__(256, 2) colsum_part_kernel(const T* __restrict__ X, int64_t ldx, int64_t n,
                                                             int64_t d, const int32_t* __restrict__ labels,
                                                             int32_t ignore, const float* __restrict__ wvec,
                                                             float* __restrict__ part, const DevScalars* sc) {
    constexpr int VEC = 16 / sizeof(T);
    __shared__ float red[8][32 * VEC];
    if (sc->status != 0) return;
    const int w = threadIdx.x >> 5, l = threadIdx.x & 31;
    const int64_t c0 = static_cast<int64_t>(blockIdx.x) * (32 * VEC) + l * VEC;
    const int64_t r0 = static_cast<int64_t>(blockIdx.y) * kRowBlock;
    const int64_t r1 = min(r0 + kRowBlock, n);
    float acc[VEC];
#pragma unroll
    for (int k = 0; k < VEC; ++k) acc[k] = 0.0f;
    const bool vec = (c0 + VEC <= d) && ((ldx % VEC) == 0);
    constexpr int UNROLL = 8;
    for (int64_t rb = r0 + w; rb < r1; rb += 8 * UNROLL) {
        uint4 raw[UNROLL];
        float wt[UNROLL];
#pragma unroll
        for (int u = 0; u < UNROLL; ++u) {
            const int64_t r = rb + 8 * u;
            wt[u] = 0.0f;
            raw[u] = make_uint4(0u, 0u, 0u, 0u);
            if (r >= r1 || c0 >= d) continue;
            float wr = 1.0f;
            if (labels) wr = (labels[r] != ignore) ? 1.0f : 0.0f;
            if (wvec) wr = wvec[r];
            wt[u] = wr;
            const T* src = X + r * ldx + c0;
            if (vec) {
                raw[u] = *reinterpret_cast<const uint4*>(src);
            } else {
                uint32_t q[4] = {0u, 0u, 0u, 0u};
#pragma unroll
                for (int k = 0; k < VEC; ++k) {
                    if (c0 + k >= d) continue;
                    if constexpr (sizeof(T) == 2)
                        q[k >> 1] |= static_cast<uint32_t>(reinterpret_cast<const uint16_t*>(src)[k]) << (16 * (k & 1));
                    else
                        q[k] = reinterpret_cast<const uint32_t*>(src)[k];
                }
                raw[u] = make_uint4(q[0], q[1], q[2], q[3]);
            }
        }
#pragma unroll
        for (int u = 0; u < UNROLL; ++u) {
            const uint32_t ws[4] = {raw[u].x, raw[u].y, raw[u].z, raw[u].w};
#pragma unroll
            for (int k = 0; k < VEC; ++k) {
                float x;
                if constexpr (sizeof(T) == 2)
                    x = __uint_as_float((k & 1) ? (ws[k >> 1] & 0xFFFF0000u) : (ws[k >> 1] << 16));
                else
                    x = __uint_as_float(ws[k]);
                acc[k] = fmaf(wt[u], x, acc[k]);
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
        part[static_cast<int64_t>(blockIdx.y) * d + c] = a;
    }
}

__global__ void __launch_bounds__(256) colsum_finish_kernel(const float* __restrict__ part, int64_t nblocks,
                                                            int64_t d, float scale, void* __restrict__ out,
                                                            int out_f32, const DevScalars* sc) {
    __shared__ float red[8][33];
    if (sc->status != 0) return;
    const int64_t j = static_cast<int64_t>(blockIdx.x) * 32 + (threadIdx.x & 31);
    const float a = fixed_order_column_sum(part, nblocks, d, j, red);
    if (threadIdx.x < 32 && j < d) st_elem(out, j, out_f32, a * scale);
}

__global__ void axpby_kernel(const float* __restrict__ s, const float* __restrict__ qh, float a, float b, int64_t V,
                             void* __restrict__ out, int out_f32, const DevScalars* sc) {
    if (sc->status != 0) return;
    const int64_t j = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x;
    if (j >= V) return;
    st_elem(out, j, out_f32, a * s[j] + b * qh[j]);
}

inline unsigned cdiv(int64_t a, int64_t b) { return static_cast<unsigned>((a + b - 1) / b); }

}  // namespace

void launch_labels_scan(const int32_t* labels, int64_t n, int64_t V, int32_t ignore, float lambda, DevScalars* sc,
                        cudaStream_t s) {
    labels_scan_kernel<<<1, 1024, 0, s>>>(labels, n, V, ignore, lambda, sc); count_launch();
}

void launch_row_stats_f32(const float* Z, int64_t ldz, int64_t n, int64_t V, float* stats, const DevScalars* sc,
                          cudaStream_t s) {
    row_stats_f32_kernel<<<cdiv(n * 32, 256), 256, 0, s>>>(Z, ldz, n, V, reinterpret_cast<float2*>(stats), sc); count_launch();
}

void launch_row_lse(const void* Z, int z_f32, int64_t ldz, int64_t n, int64_t V, const float* stats, int64_t ntiles,
                    const int32_t* labels, int32_t ignore, float* lse, float* ce, const DevScalars* sc,
                    cudaStream_t s) {
    row_lse_kernel<<<cdiv(n * 32, 256), 256, 0, s>>>(Z, z_f32, ldz, n, V, reinterpret_cast<const float2*>(stats),
                                                      ntiles, labels, ignore, lse, ce, sc); count_launch();
}

void launch_residual(void* Z, int z_f32, int64_t ldz, int64_t n, int64_t V, const float* lse, const int32_t* labels,
                     int32_t ignore, float* colpart, const DevScalars* sc, cudaStream_t s) {
    if (z_f32) {
        dim3 grid(cdiv(ldz, 256 * 4), static_cast<unsigned>(resid_blocks(n)));
        residual_kernel<float, 4><<<grid, 256, 0, s>>>(static_cast<float*>(Z), ldz, n, V, lse, labels, ignore,
                                                       colpart, sc); count_launch();
    } else {
        dim3 grid(cdiv(ldz, 256 * 8), static_cast<unsigned>(resid_blocks(n)));
        residual_kernel<__nv_bfloat16, 8><<<grid, 256, 0, s>>>(static_cast<__nv_bfloat16*>(Z), ldz, n, V, lse,
                                                               labels, ignore, colpart, sc); count_launch();
    }
}

void launch_finish_sq(const float* colpart, int64_t nblocks, int64_t V, float beta1, float inv_bc1, float* q,
                      float* s_out, float* qhat, DevScalars* sc, cudaStream_t s) {
    finish_sq_kernel<<<cdiv(V, 32), 256, 0, s>>>(colpart, nblocks, V, beta1, inv_bc1, q, s_out, qhat, sc); count_launch();
}

void launch_scalars(const float* ce, int64_t n, const float* s_vec, int64_t V, DevScalars* sc, cudaStream_t s) {
    scalars_kernel<<<1, 1024, 0, s>>>(ce, n, s_vec, V, sc); count_launch();
}

void launch_colsum(const void* X, int x_f32, int64_t ldx, int64_t n, int64_t d, const int32_t* labels,
                   int32_t ignore, const float* wvec, float scale, float* part, void* out, int out_f32,
                   const DevScalars* sc, cudaStream_t s) {
    const int64_t nb = row_blocks(n);
    if (x_f32) {
        dim3 grid(cdiv(d, 128), static_cast<unsigned>(nb));
        colsum_part_kernel<float><<<grid, 256, 0, s>>>(static_cast<const float*>(X), ldx, n, d, labels, ignore, wvec,
                                                       part, sc);
    } else {
        dim3 grid(cdiv(d, 256), static_cast<unsigned>(nb));
        colsum_part_kernel<__nv_bfloat16><<<grid, 256, 0, s>>>(static_cast<const __nv_bfloat16*>(X), ldx, n, d,
                                                               labels, ignore, wvec, part, sc);
    }
    count_launch();
    colsum_finish_kernel<<<cdiv(d, 32), 256, 0, s>>>(part, nb, d, scale, out, out_f32, sc); count_launch();
}

void launch_axpby(const float* s_vec, const float* qhat, float a, float b, int64_t V, void* out, int out_f32,
                  const DevScalars* sc, cudaStream_t s) {
    axpby_kernel<<<cdiv(V, 256), 256, 0, s>>>(s_vec, qhat, a, b, V, out, out_f32, sc); count_launch();
}

}  // namespace bom
