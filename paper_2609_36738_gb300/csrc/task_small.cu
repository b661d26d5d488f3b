// Task-space pass of a small step in one cluster launch.
//
// For small batches and output spaces (the classification settings: batch 32
// x 10 classes, batch 256 x 1000 classes) the task-space part of Algorithm 1
// is a handful of tiny reductions, and as separate kernels each costs its
// launch and pipeline fill rather than its work.  One cluster of 16 CTAs (8
// where the device allows no larger cluster or the pass is a few dozen rows)
// does all of it, with the cross-CTA sums in distributed shared memory (added in
// rank order, so the result is deterministic):
//   phase 1 (rows split over the CTAs): label check and N_t, the row
//           log-sum-exp and CE from the logits, r_i = softmax(z_i) - onehot(y_i)
//           written over Z (0 on ignored rows), column sums of R and of
//           1_{I_t} H over the CTA's rows;
//   phase 2 (vocabulary columns split): s_t = N_t^-1 sum_i r_i,
//           q_t = beta1 q_{t-1} + (1-beta1) s_t, qhat_t = q_t / (1-beta1^t)
//           (Section 3.2), the head bias numerator a s + b qhat, the step
//           scalars (N_t, cotangent coefficients, loss, lr and both bias
//           corrections) and c = colsum_{I_t}(H);
//   phase 3 (the CTA's vocabulary rows of W): partial sums of W^T qhat;
//   phase 4 (d split): w = W^T qhat, ||s_t||.
// Error precedence follows the multi-kernel path: a bad label or N_t = 0
// first, then a device step counter below 1, then non-finite logits; q and
// every output of phase 2 on are written only when no error is latched.
#include <cooperative_groups.h>

#include <atomic>

#include "kernels.h"

namespace bom {

namespace {

namespace cg = cooperative_groups;

// Cluster sizes: 16 CTAs where the device allows a cluster of that size
// (non-portable), else the portable 8; the per-CTA rows, vocabulary and d
// slices, and with them the serial rounds of loads of each phase, halve with 16.
constexpr int kSmallClusterMax = 16;
constexpr int kSmallClusterMin = 8;
// A pass whose logits, head inputs and head weights fit in one CTA's shared
// memory together (the tiny classifier: 32 x 10 logits, 32 x 128 inputs) runs
// from there (task_tiny_kernel): one round of loads, then every phase at
// shared-memory latency.
constexpr int64_t kTinyStageFloats = 16384;
constexpr int kSmallThreads = 1024;
// Row-group partials of the chunked column sums: RG * dm <= 1024 * 8 floats
// (RG = 1024 / (dm / elements per 16-byte word), or 1).
constexpr int kSmallPart = 8192;

struct TaskSmallArgs {
    const void* Z;
    int64_t ldz;
    const int32_t* labels;
    int64_t n, V;
    int32_t ignore;
    float lambda, beta1;
    const void* H;      // head input [n, dm] (row pitch dm)
    const void* W;      // head weight [V, dm]
    int64_t dm;
    float* q;
    float* s_out;
    float* qhat;
    float* lse;
    float* cvec;
    float* wvec;
    void* hb_out;       // head bias numerator hb_a s + hb_b qhat, or NULL
    int hb_f32;
    float hb_a, hb_b;
    StepScalarsIn st;
    DevScalars* sc;
};

__device__ __forceinline__ float warp_sum_f(float v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    return v;
}
__device__ __forceinline__ float warp_max_f(float v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
    return v;
}

template <typename T>
__device__ __forceinline__ float ld_t(const void* p, int64_t i) {
    if constexpr (sizeof(T) == 4)
        return static_cast<const float*>(p)[i];
    else
        return __bfloat162float(static_cast<const __nv_bfloat16*>(p)[i]);
}
template <typename T>
__device__ __forceinline__ void st_t(void* p, int64_t i, float v) {
    if constexpr (sizeof(T) == 4)
        static_cast<float*>(p)[i] = v;
    else
        static_cast<__nv_bfloat16*>(p)[i] = __float2bfloat16_rn(v);
}
// Element e of a 16-byte word holding 16 / sizeof(T) values.
template <typename T>
__device__ __forceinline__ float word_at(const uint4& w, int e) {
    const uint32_t x = (e * static_cast<int>(sizeof(T)) / 4) == 0   ? w.x
                       : (e * static_cast<int>(sizeof(T)) / 4) == 1 ? w.y
                       : (e * static_cast<int>(sizeof(T)) / 4) == 2 ? w.z
                                                                     : w.w;
    if constexpr (sizeof(T) == 4)
        return __uint_as_float(x);
    else
        return __uint_as_float((e & 1) ? (x & 0xFFFF0000u) : (x << 16));
}

// part[g * dm + k] = sum over rows j = j0 + g, j0 + g + RG, ... < j1 of
// wt(j) * X[j, k], for g < RG row groups: thread (kc, g) reads its rows' word
// kc of 16 bytes, four rows in flight.  RG * KC <= 1024 (RG = 1024 / KC).
// `vec` selects 16-byte words (rows 16-byte aligned, dm a multiple of the
// word) or single elements.
template <typename T, class Wt>
__device__ __forceinline__ void colsum_tile(const void* X, int64_t dm, int64_t j0, int64_t j1, bool vec, Wt wt,
                                            float* part, int RG) {
    const int EPC = vec ? 16 / static_cast<int>(sizeof(T)) : 1;
    const int64_t KC = (dm + EPC - 1) / EPC;
    for (int64_t idx = threadIdx.x; idx < KC * RG; idx += kSmallThreads) {
        const int64_t kc = idx % KC;
        const int g = static_cast<int>(idx / KC);
        float acc[8];
#pragma unroll
        for (int e = 0; e < 8; ++e) acc[e] = 0.0f;
        int64_t j = j0 + g;
        if (vec) {
            // batches of four rows, the last one predicated (a missing row
            // reads nothing and has weight 0): every batch has its four loads
            // in flight, and the rows are still added in increasing order
            const T* base = static_cast<const T*>(X) + kc * EPC;
            for (; j < j1; j += 4 * RG) {
                uint4 w[4];
                float f[4];
#pragma unroll
                for (int u = 0; u < 4; ++u) {
                    const int64_t jj = j + u * RG;
                    w[u] = jj < j1 ? __ldg(reinterpret_cast<const uint4*>(base + jj * dm)) : make_uint4(0u, 0u, 0u, 0u);
                    f[u] = jj < j1 ? wt(jj) : 0.0f;
                }
#pragma unroll
                for (int u = 0; u < 4; ++u)
                    if (j + u * RG < j1)
#pragma unroll
                        for (int e = 0; e < 8; ++e)
                            if (e < EPC) acc[e] = fmaf(f[u], word_at<T>(w[u], e), acc[e]);
            }
        } else {
            for (; j < j1; j += RG) acc[0] = fmaf(wt(j), ld_t<T>(X, j * dm + kc), acc[0]);
        }
        for (int e = 0; e < EPC; ++e)
            if (kc * EPC + e < dm) part[g * dm + kc * EPC + e] = acc[e];
    }
}

// Shared memory of one CTA (floats unless noted), sized by the host:
//   colp[V]     column sums of R over the CTA's rows
//   cp[dm]      column sums of 1_{I_t} H over the CTA's rows
//   wp[dm]      partial W^T qhat over the CTA's vocabulary rows
//   part[8192]  row-group partials of the two chunked column sums
//   qh[vs]      qhat of the CTA's vocabulary slice
//   lse_s[rp], lab_s[rp] (int)   the CTA's rows
//   per-warp CE, N_t, bad-label and non-finite counts [4][32], totals
template <typename T, int C>
__global__ void __launch_bounds__(kSmallThreads, 1) task_small_kernel(const TaskSmallArgs a) {
    pdl_enter();
    cg::cluster_group cl = cg::this_cluster();
    constexpr int EPC = 16 / static_cast<int>(sizeof(T));
    const int c = static_cast<int>(cl.block_rank());
    const int64_t V = a.V, dm = a.dm, n = a.n;
    const int64_t rp = (n + C - 1) / C;             // rows per CTA
    const int64_t vs = (V + C - 1) / C;             // vocabulary columns per CTA
    const int64_t ds = (dm + C - 1) / C;            // d columns per CTA
    extern __shared__ float sm[];
    float* colp = sm;
    float* cp = colp + V;
    float* wp = cp + dm;
    float* part = wp + dm;
    float* qh = part + kSmallPart;
    float* lse_s = qh + vs;
    int* lab_s = reinterpret_cast<int*>(lse_s + rp);
    float* wce = reinterpret_cast<float*>(lab_s + rp);
    int* wnt = reinterpret_cast<int*>(wce + 32);
    int* wbad = wnt + 32;
    int* wnf = wbad + 32;
    float* tot_f = reinterpret_cast<float*>(wnf + 32);   // [0] CE sum, [1] sum s^2 of the slice
    int* tot_i = reinterpret_cast<int*>(tot_f + 2);      // [0] N_t, [1] bad, [2] non-finite

    const int tid = threadIdx.x, w = tid >> 5, l = tid & 31;
    // the device step counter and learning rate are loaded now and kept
    // after phase 1a, so that their latency is off the single-thread chain of
    // phase 2
    __shared__ int64_t s_t;
    __shared__ float s_lr;
    int64_t t_ld = 1;
    float lr_ld = a.st.lr;
    if (tid == 0) {
        if (a.st.t_dev != nullptr) t_ld = __ldcg(a.st.t_dev);
        if (a.st.lr_dev != nullptr) lr_ld = __ldcg(a.st.lr_dev);
    }
    const bool live = a.sc->status == 0;
    const int64_t r0 = c * rp < n ? c * rp : n;
    const int64_t r1 = r0 + rp < n ? r0 + rp : n;
    // rows of H and W start on 16 bytes when dm fills whole words
    const bool hw_vec = (dm % EPC) == 0;
    const int64_t KC = hw_vec ? dm / EPC : dm;
    const int RG = static_cast<int>(kSmallThreads / KC > 0 ? kSmallThreads / KC : 1);

    // ---- phase 1a: one warp per row, the row read as 16-byte words (Z rows
    // are padded to whole 128-byte lines), four words in flight per lane
    float ce_w = 0.0f;
    int nt_w = 0, bad_w = 0, nf_w = 0;
    {   // read whatever the status word says (it only gates the writes), so
        // that its latency overlaps the row reads
        const int64_t nw = (V + EPC - 1) / EPC;
        for (int64_t r = r0 + w; r < r1; r += kSmallThreads / 32) {
            const int32_t y = a.labels[r];
            const bool sup = y != a.ignore;
            const bool ok_y = sup && y >= 0 && y < V;
            const T* zr = static_cast<const T*>(a.Z) + r * a.ldz;
            float m = -INFINITY;
            if (nw <= 128) {
                // the whole row in registers (four words per lane): one read
                // for the maximum, the sum and z_y
                uint4 wd[4];
#pragma unroll
                for (int u = 0; u < 4; ++u)
                    wd[u] = l + 32 * u < nw ? *reinterpret_cast<const uint4*>(zr + (l + 32 * u) * EPC)
                                            : make_uint4(0u, 0u, 0u, 0u);
                if constexpr (sizeof(T) == 2) {
                    // packed maximum on the raw bf16 pairs (columns past V
                    // masked to -inf), so the unpacked values live only in
                    // the sum below
                    uint32_t mm = 0xFF80FF80u;
#pragma unroll
                    for (int u = 0; u < 4; ++u) {
                        const int64_t c0 = (l + 32 * u) * EPC;
                        const uint32_t x4[4] = {wd[u].x, wd[u].y, wd[u].z, wd[u].w};
#pragma unroll
                        for (int q2 = 0; q2 < 4; ++q2) {
                            const int64_t cc = c0 + 2 * q2;
                            const uint32_t lo = cc < V ? (x4[q2] & 0xFFFFu) : 0xFF80u;
                            const uint32_t hi = cc + 1 < V ? (x4[q2] & 0xFFFF0000u) : 0xFF800000u;
                            mm = max_bf16x2(mm, lo | hi);
                        }
                    }
                    m = fmaxf(bf16_lo(mm), bf16_hi(mm));
                } else {
#pragma unroll
                    for (int u = 0; u < 4; ++u)
#pragma unroll
                        for (int e = 0; e < EPC; ++e)
                            if ((l + 32 * u) * EPC + e < V) m = fmaxf(m, word_at<T>(wd[u], e));
                }
                m = warp_max_f(m);
                float s = 0.0f;
#pragma unroll
                for (int u = 0; u < 4; ++u)
#pragma unroll
                    for (int e = 0; e < EPC; ++e)
                        if ((l + 32 * u) * EPC + e < V) s += expf(word_at<T>(wd[u], e) - m);
                s = warp_sum_f(s);
                // z_y from the lane holding word y / EPC (ok_y is the same on every lane)
                float zy = 0.0f;
                if (ok_y) {
                    const int kw = y / EPC, ey = y - kw * EPC, su = kw >> 5;
                    float cand = 0.0f;
#pragma unroll
                    for (int u = 0; u < 4; ++u)
                        if (u == su) cand = word_at<T>(wd[u], ey);
                    zy = __shfl_sync(0xffffffffu, cand, kw & 31);
                }
                if (l == 0) {
                    const float L = m + logf(s);
                    lse_s[r - r0] = L;
                    lab_s[r - r0] = ok_y ? y : -1;
                    if (live) a.lse[r] = L;
                    if (sup && !ok_y) ++bad_w;
                    if (ok_y) {
                        ++nt_w;
                        ce_w += L - zy;
                    }
                    if (!isfinite(L) || (ok_y && !isfinite(zy))) ++nf_w;
                }
                continue;
            }
            for (int64_t b = l; b < nw; b += 128) {
                uint4 wd[4];
#pragma unroll
                for (int u = 0; u < 4; ++u)
                    if (b + 32 * u < nw) wd[u] = *reinterpret_cast<const uint4*>(zr + (b + 32 * u) * EPC);
#pragma unroll
                for (int u = 0; u < 4; ++u)
                    if (b + 32 * u < nw)
#pragma unroll
                        for (int e = 0; e < EPC; ++e)
                            if ((b + 32 * u) * EPC + e < V) m = fmaxf(m, word_at<T>(wd[u], e));
            }
            m = warp_max_f(m);
            float s = 0.0f;
            for (int64_t b = l; b < nw; b += 128) {
                uint4 wd[4];
#pragma unroll
                for (int u = 0; u < 4; ++u)
                    if (b + 32 * u < nw) wd[u] = *reinterpret_cast<const uint4*>(zr + (b + 32 * u) * EPC);
#pragma unroll
                for (int u = 0; u < 4; ++u)
                    if (b + 32 * u < nw)
#pragma unroll
                        for (int e = 0; e < EPC; ++e)
                            if ((b + 32 * u) * EPC + e < V) s += expf(word_at<T>(wd[u], e) - m);
            }
            s = warp_sum_f(s);
            if (l == 0) {
                const float L = m + logf(s);
                lse_s[r - r0] = L;
                lab_s[r - r0] = ok_y ? y : -1;
                if (live) a.lse[r] = L;
                const float zy = ok_y ? ld_t<T>(a.Z, r * a.ldz + y) : 0.0f;
                if (sup && !ok_y) ++bad_w;
                if (ok_y) {
                    ++nt_w;
                    ce_w += L - zy;
                }
                if (!isfinite(L) || (ok_y && !isfinite(zy))) ++nf_w;
            }
        }
    }
    if (l == 0) {
        wce[w] = ce_w;
        wnt[w] = nt_w;
        wbad[w] = bad_w;
        wnf[w] = nf_w;
    }
    if (tid == 0) {
        s_t = t_ld;
        s_lr = lr_ld;
    }
    __syncthreads();
    if (tid == 0) {
        float ce = 0.0f;
        int nt = 0, bad = 0, nf = 0;
        for (int k = 0; k < kSmallThreads / 32; ++k) {
            ce += wce[k];
            nt += wnt[k];
            bad += wbad[k];
            nf += wnf[k];
        }
        tot_f[0] = ce;
        tot_i[0] = nt;
        tot_i[1] = bad;
        tot_i[2] = nf;
    }
    // ---- phase 1b: one thread per column, the CTA's rows in order, eight in flight
    if (live) {
        for (int64_t j = tid; j < V; j += kSmallThreads) {
            float acc = 0.0f;
            for (int64_t rb = r0; rb < r1; rb += 8) {
                float z[8];
#pragma unroll
                for (int u = 0; u < 8; ++u) z[u] = rb + u < r1 ? ld_t<T>(a.Z, (rb + u) * a.ldz + j) : 0.0f;
#pragma unroll
                for (int u = 0; u < 8; ++u) {
                    const int64_t r = rb + u;
                    if (r >= r1) break;
                    const int y = lab_s[r - r0];
                    float p = 0.0f;
                    if (y >= 0) {
                        p = expf(z[u] - lse_s[r - r0]);
                        if (j == y) p -= 1.0f;
                    }
                    st_t<T>(const_cast<void*>(a.Z), r * a.ldz + j, p);
                    acc += p;
                }
            }
            colp[j] = acc;
        }
        // c over the CTA's rows: 1_{I_t} H, in row groups, then the groups in order
        colsum_tile<T>(a.H, dm, r0, r1, hw_vec, [&](int64_t r) { return lab_s[r - r0] >= 0 ? 1.0f : 0.0f; },
                       part, RG);
        __syncthreads();
        for (int64_t k = tid; k < dm; k += kSmallThreads) {
            float acc = 0.0f;
            for (int g = 0; g < RG; ++g) acc += part[g * dm + k];
            cp[k] = acc;
        }
    }
    cl.sync();

    // ---- phase 2: totals, status, s / q / qhat of the CTA's vocabulary slice.
    // The two bias corrections (fp64 products) are formed by two other
    // threads at the same time as the totals.
    __shared__ int s_code, s_nt;
    __shared__ float s_inv_nt, s_bc1, s_bc2, s_tot_ce;
    const bool t_bad = a.st.t_dev != nullptr && s_t < 1;
    if (tid == 32) s_bc1 = (a.st.t_dev != nullptr && !t_bad) ? inv_bias_correction(a.st.beta1, s_t) : a.st.inv_bc1;
    if (tid == 64) s_bc2 = (a.st.t_dev != nullptr && !t_bad) ? inv_bias_correction(a.st.beta2, s_t) : a.st.inv_bc2;
    if (tid == 0) {
        float ce = 0.0f;
        int nt = 0, bad = 0, nf = 0;
#pragma unroll
        for (int cc = 0; cc < C; ++cc) {
            const float* tf = cl.map_shared_rank(tot_f, cc);
            const int* ti = cl.map_shared_rank(tot_i, cc);
            ce += tf[0];
            nt += ti[0];
            bad += ti[1];
            nf += ti[2];
        }
        int code = live ? 0 : -1;
        if (live) {
            if (bad > 0)
                code = BOM_ELABEL;
            else if (nt == 0)
                code = BOM_EEMPTY;
            else if (t_bad)
                code = BOM_EINVAL;
            else if (nf > 0)
                code = BOM_ENONFINITE;
        }
        const float inv = nt > 0 ? 1.0f / static_cast<float>(nt) : 0.0f;
        s_code = code;
        s_nt = nt;
        s_inv_nt = inv;
        s_tot_ce = ce;
    }
    __syncthreads();
    if (tid == 0 && c == 0 && live) {
        const int code = s_code, nt = s_nt;
        const float inv = s_inv_nt, ce = s_tot_ce;
        {
            DevScalars* sc = a.sc;
            if (code > 0) latch_status(sc, code);
            sc->n_t = nt;
            sc->inv_nt = inv;
            sc->coef_r[0] = (1.0f - a.lambda) * inv;
            sc->coef_q[0] = a.lambda * inv;
            sc->coef_r[1] = inv;
            sc->coef_q[1] = 0.0f;
            sc->coef_r[2] = 0.0f;
            sc->coef_q[2] = inv;
            sc->coef_r[3] = 0.0f;
            sc->coef_q[3] = inv;
            sc->lr = s_lr;
            sc->inv_bc1 = s_bc1;
            sc->inv_bc2 = s_bc2;
            sc->loss = ce * inv;
            sc->s_norm = 0.0f;
            sc->r_norm_mean = 0.0f;
        }
    }
    __syncthreads();
    const bool ok = s_code == 0;
    const int64_t j0 = c * vs < V ? c * vs : V;
    const int64_t j1 = j0 + vs < V ? j0 + vs : V;
    const int64_t k0 = c * ds < dm ? c * ds : dm;
    const int64_t k1 = k0 + ds < dm ? k0 + ds : dm;
    float ss = 0.0f;
    if (ok) {
        const float inv = s_inv_nt, bc1 = s_bc1;
        for (int64_t j = j0 + tid; j < j1; j += kSmallThreads) {
            float pv[C];
#pragma unroll
            for (int cc = 0; cc < C; ++cc) pv[cc] = cl.map_shared_rank(colp, cc)[j];
            float acc = 0.0f;
#pragma unroll
            for (int cc = 0; cc < C; ++cc) acc += pv[cc];
            const float s = acc * inv;
            const float qn = a.beta1 * a.q[j] + (1.0f - a.beta1) * s;
            const float qhat = qn * bc1;
            a.q[j] = qn;
            a.s_out[j] = s;
            a.qhat[j] = qhat;
            qh[j - j0] = qhat;
            ss += s * s;
            if (a.hb_out) st_elem(a.hb_out, j, a.hb_f32, a.hb_a * s + a.hb_b * qhat);
        }
        for (int64_t k = k0 + tid; k < k1; k += kSmallThreads) {
            float pv[C];
#pragma unroll
            for (int cc = 0; cc < C; ++cc) pv[cc] = cl.map_shared_rank(cp, cc)[k];
            float acc = 0.0f;
#pragma unroll
            for (int cc = 0; cc < C; ++cc) acc += pv[cc];
            a.cvec[k] = acc;
        }
    }
    ss = warp_sum_f(ss);
    if (l == 0) wce[w] = ss;
    __syncthreads();
    if (tid == 0) {
        float t = 0.0f;
        for (int k = 0; k < kSmallThreads / 32; ++k) t += wce[k];
        tot_f[1] = t;
    }
    // ---- phase 3: partial W^T qhat over the CTA's vocabulary rows (row
    // groups of 16-byte words, then the groups in order)
    if (ok) {
        colsum_tile<T>(a.W, dm, j0, j1, hw_vec, [&](int64_t j) { return qh[j - j0]; }, part, RG);
        __syncthreads();
        for (int64_t k = tid; k < dm; k += kSmallThreads) {
            float acc = 0.0f;
            for (int g = 0; g < RG; ++g) acc += part[g * dm + k];
            wp[k] = acc;
        }
    }
    cl.sync();
    // ---- phase 4: w = W^T qhat over the d slice, ||s_t||
    if (ok) {
        for (int64_t k = k0 + tid; k < k1; k += kSmallThreads) {
            float pv[C];
#pragma unroll
            for (int cc = 0; cc < C; ++cc) pv[cc] = cl.map_shared_rank(wp, cc)[k];
            float acc = 0.0f;
#pragma unroll
            for (int cc = 0; cc < C; ++cc) acc += pv[cc];
            a.wvec[k] = acc;
        }
        if (c == 0 && tid == 0) {
            float t = 0.0f;
#pragma unroll
            for (int cc = 0; cc < C; ++cc) t += cl.map_shared_rank(tot_f, cc)[1];
            a.sc->s_norm = sqrtf(t);
        }
    }
    cl.sync();   // no CTA leaves while another still reads its shared memory
}

// The same pass for tiny sizes, in one CTA from shared memory: Z, H and W
// are read once into shared memory (fp32), then the phases of the cluster
// kernel run on those copies with the same outputs and the same error
// precedence; R still goes to Z in global memory for the backward GEMMs.
// Shared memory (floats): zs[n V], hs[n dm], ws[V dm], lse_s[n], lab_s[n]
// (int), colp[V], qh[V], cs[dm].
template <typename T>
__global__ void __launch_bounds__(kSmallThreads, 1) task_tiny_kernel(const TaskSmallArgs a) {
    pdl_enter();
    const int64_t V = a.V, dm = a.dm, n = a.n;
    extern __shared__ float sm[];
    float* zs = sm;
    float* hs = zs + n * V;
    float* ws = hs + n * dm;
    float* lse_s = ws + V * dm;
    int* lab_s = reinterpret_cast<int*>(lse_s + n);
    float* colp = reinterpret_cast<float*>(lab_s + n);
    float* qh = colp + V;
    float* cs = qh + V;
    __shared__ float wf[32];
    __shared__ int wi[3][32];
    __shared__ int s_code, s_nt;
    __shared__ float s_inv_nt, s_bc1, s_bc2, s_ce, s_ss;
    __shared__ int64_t s_t;
    const int tid = threadIdx.x, w = tid >> 5, l = tid & 31;

    // the device step counter and learning rate (thread 0 reads them; the
    // counter goes to shared memory for the two bias-correction threads)
    int64_t t_ld = 1;
    float lr_ld = a.st.lr;
    if (tid == 0) {
        if (a.st.t_dev != nullptr) t_ld = __ldcg(a.st.t_dev);
        if (a.st.lr_dev != nullptr) lr_ld = __ldcg(a.st.lr_dev);
        s_t = t_ld;
    }
    const bool live = a.sc->status == 0;
    // stage Z, H and W: one index space, eight loads in flight per thread
    {
        const int64_t e0 = n * V, e1 = e0 + n * dm, e2 = e1 + V * dm;
        for (int64_t base = 0; base < e2; base += 8 * kSmallThreads) {
            float v[8];
#pragma unroll
            for (int u = 0; u < 8; ++u) {
                const int64_t i = base + u * kSmallThreads + tid;
                if (i < e0)
                    v[u] = ld_t<T>(a.Z, (i / V) * a.ldz + i % V);
                else if (i < e1)
                    v[u] = ld_t<T>(a.H, i - e0);
                else if (i < e2)
                    v[u] = ld_t<T>(a.W, i - e1);
                else
                    v[u] = 0.0f;
            }
#pragma unroll
            for (int u = 0; u < 8; ++u) {
                const int64_t i = base + u * kSmallThreads + tid;
                if (i < e2) sm[i] = v[u];
            }
        }
    }
    __syncthreads();

    // rows: one warp per row, log-sum-exp, CE, label check
    float ce_w = 0.0f;
    int nt_w = 0, bad_w = 0, nf_w = 0;
    for (int64_t r = w; r < n; r += kSmallThreads / 32) {
        const int32_t y = a.labels[r];
        const bool sup = y != a.ignore;
        const bool ok_y = sup && y >= 0 && y < V;
        const float* zr = zs + r * V;
        float m = -INFINITY;
        for (int64_t j = l; j < V; j += 32) m = fmaxf(m, zr[j]);
        m = warp_max_f(m);
        float sum = 0.0f;
        for (int64_t j = l; j < V; j += 32) sum += expf(zr[j] - m);
        sum = warp_sum_f(sum);
        if (l == 0) {
            const float L = m + logf(sum);
            const float zy = ok_y ? zr[y] : 0.0f;
            lse_s[r] = L;
            lab_s[r] = ok_y ? y : -1;
            if (live) a.lse[r] = L;
            if (sup && !ok_y) ++bad_w;
            if (ok_y) {
                ++nt_w;
                ce_w += L - zy;
            }
            if (!isfinite(L) || (ok_y && !isfinite(zy))) ++nf_w;
        }
    }
    if (l == 0) {
        wf[w] = ce_w;
        wi[0][w] = nt_w;
        wi[1][w] = bad_w;
        wi[2][w] = nf_w;
    }
    __syncthreads();
    // R over Z (0 on rows outside I_t), kept in zs for the column sums
    for (int64_t i = tid; i < n * V; i += kSmallThreads) {
        const int64_t r = i / V, j = i % V;
        const int y = lab_s[r];
        float pr = 0.0f;
        if (y >= 0) {
            pr = expf(zs[i] - lse_s[r]);
            if (j == y) pr -= 1.0f;
        }
        zs[i] = pr;
        if (live) st_t<T>(const_cast<void*>(a.Z), r * a.ldz + j, pr);
    }
    if (tid == 0) {
        float ce = 0.0f;
        int nt = 0, bad = 0, nf = 0;
        for (int k = 0; k < kSmallThreads / 32; ++k) {
            ce += wf[k];
            nt += wi[0][k];
            bad += wi[1][k];
            nf += wi[2][k];
        }
        const bool t_bad = a.st.t_dev != nullptr && t_ld < 1;
        int code = live ? 0 : -1;
        if (live) {
            if (bad > 0)
                code = BOM_ELABEL;
            else if (nt == 0)
                code = BOM_EEMPTY;
            else if (t_bad)
                code = BOM_EINVAL;
            else if (nf > 0)
                code = BOM_ENONFINITE;
        }
        s_code = code;
        s_nt = nt;
        s_inv_nt = nt > 0 ? 1.0f / static_cast<float>(nt) : 0.0f;
        s_ce = ce;
    }
    // the two fp64 bias corrections beside it
    if (tid == 32)
        s_bc1 = (a.st.t_dev != nullptr && s_t >= 1) ? inv_bias_correction(a.st.beta1, s_t) : a.st.inv_bc1;
    if (tid == 64)
        s_bc2 = (a.st.t_dev != nullptr && s_t >= 1) ? inv_bias_correction(a.st.beta2, s_t) : a.st.inv_bc2;
    __syncthreads();
    // column sums of R and of 1_{I_t} H, rows in order
    for (int64_t j = tid; j < V; j += kSmallThreads) {
        float acc = 0.0f;
        for (int64_t r = 0; r < n; ++r) acc += zs[r * V + j];
        colp[j] = acc;
    }
    for (int64_t k = tid; k < dm; k += kSmallThreads) {
        float acc = 0.0f;
        for (int64_t r = 0; r < n; ++r)
            if (lab_s[r] >= 0) acc += hs[r * dm + k];
        cs[k] = acc;
    }
    if (tid == 0 && live) {
        DevScalars* sc = a.sc;
        const int code = s_code;
        const float inv = s_inv_nt;
        if (code > 0) latch_status(sc, code);
        sc->n_t = s_nt;
        sc->inv_nt = inv;
        sc->coef_r[0] = (1.0f - a.lambda) * inv;
        sc->coef_q[0] = a.lambda * inv;
        sc->coef_r[1] = inv;
        sc->coef_q[1] = 0.0f;
        sc->coef_r[2] = 0.0f;
        sc->coef_q[2] = inv;
        sc->coef_r[3] = 0.0f;
        sc->coef_q[3] = inv;
        sc->lr = lr_ld;
        sc->inv_bc1 = s_bc1;
        sc->inv_bc2 = s_bc2;
        sc->loss = s_ce * inv;
        sc->s_norm = 0.0f;
        sc->r_norm_mean = 0.0f;
    }
    __syncthreads();
    const bool ok = s_code == 0;
    // s_t, q_t, qhat_t (Section 3.2), the head bias numerator, c
    float ss = 0.0f;
    if (ok) {
        const float inv = s_inv_nt, bc1 = s_bc1;
        for (int64_t j = tid; j < V; j += kSmallThreads) {
            const float sv = colp[j] * inv;
            const float qn = a.beta1 * a.q[j] + (1.0f - a.beta1) * sv;
            const float qhat = qn * bc1;
            a.q[j] = qn;
            a.s_out[j] = sv;
            a.qhat[j] = qhat;
            qh[j] = qhat;
            ss += sv * sv;
            if (a.hb_out) st_elem(a.hb_out, j, a.hb_f32, a.hb_a * sv + a.hb_b * qhat);
        }
        for (int64_t k = tid; k < dm; k += kSmallThreads) a.cvec[k] = cs[k];
    }
    ss = warp_sum_f(ss);
    if (l == 0) wf[w] = ss;
    __syncthreads();
    if (tid == 0) {
        float t = 0.0f;
        for (int k = 0; k < kSmallThreads / 32; ++k) t += wf[k];
        s_ss = t;
    }
    // w = W^T qhat, vocabulary rows in order
    if (ok)
        for (int64_t k = tid; k < dm; k += kSmallThreads) {
            float acc = 0.0f;
            for (int64_t j = 0; j < V; ++j) acc = fmaf(qh[j], ws[j * dm + k], acc);
            a.wvec[k] = acc;
        }
    if (ok && tid == 0) a.sc->s_norm = sqrtf(s_ss);
}

size_t task_tiny_smem(int64_t n, int64_t V, int64_t dm) {
    return static_cast<size_t>(4 * (n * V + n * dm + V * dm + 2 * n + 2 * V + dm) + 64);
}

bool tiny_fits(int64_t n, int64_t V, int64_t dm) {
    return n * V + n * dm + V * dm <= kTinyStageFloats && n <= 1024 && V <= 1024 && dm <= 1024;
}

size_t task_small_smem(int64_t n, int64_t V, int64_t dm, int C) {
    const int64_t rp = (n + C - 1) / C;
    const int64_t vs = (V + C - 1) / C;
    return static_cast<size_t>(4 * (V + 2 * dm + kSmallPart + vs + 2 * rp + 4 * 32 + 2 + 3) + 64);
}

cudaLaunchConfig_t small_cfg(cudaLaunchAttribute (&at)[2], int C, size_t smem, cudaStream_t s) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(C);
    cfg.blockDim = dim3(kSmallThreads);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = s;
    at[0].id = cudaLaunchAttributeClusterDimension;
    at[0].val.clusterDim.x = C;
    at[0].val.clusterDim.y = 1;
    at[0].val.clusterDim.z = 1;
    at[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    at[1].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = at;
    cfg.numAttrs = 2;
    return cfg;
}

// Whether a cluster of C CTAs of the kernel at its largest shared-memory
// size fits on the current device (the attributes are per-device settings).
template <typename T, int C>
bool cluster_fits() {
    const size_t smem = task_small_smem(kTaskSmallMaxRows, kTaskSmallMaxV, kTaskSmallMaxD, C);
    bool ok = cudaFuncSetAttribute(task_small_kernel<T, C>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                   static_cast<int>(smem)) == cudaSuccess;
    if (ok && C > 8)
        ok = cudaFuncSetAttribute(task_small_kernel<T, C>, cudaFuncAttributeNonPortableClusterSizeAllowed, 1) ==
             cudaSuccess;
    if (ok) {
        cudaLaunchAttribute at[2];
        cudaLaunchConfig_t cfg = small_cfg(at, C, smem, nullptr);
        int nc = 0;
        ok = cudaOccupancyMaxActiveClusters(&nc, task_small_kernel<T, C>, &cfg) == cudaSuccess && nc >= 1;
    }
    cudaGetLastError();
    return ok;
}

// Per device, found once: the largest cluster size the path can run with
// (0: the path is not usable).
template <typename T>
int small_cluster() {
    constexpr int kMaxDev = 64;
    static std::atomic<int> state[kMaxDev];   // 0 unknown, -1 not usable, else the cluster size
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDev) {
        cudaGetLastError();
        return 0;
    }
    int st = state[dev].load(std::memory_order_relaxed);
    if (st == 0) {
        // every size is set up: a launch may take a smaller one
        // the tiny pass: at most kTinyStageFloats staged and n, V, d <= 1024
        const size_t tiny_smem = 4 * (kTinyStageFloats + 5 * 1024) + 64;
        const bool tiny_ok = cudaFuncSetAttribute(task_tiny_kernel<T>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                                  static_cast<int>(tiny_smem)) == cudaSuccess;
        cudaGetLastError();
        const bool fits_min = cluster_fits<T, kSmallClusterMin>() && tiny_ok;
        const bool fits_max = fits_min && cluster_fits<T, kSmallClusterMax>();
        st = fits_max ? kSmallClusterMax : fits_min ? kSmallClusterMin : -1;
        state[dev].store(st, std::memory_order_relaxed);
    }
    return st > 0 ? st : 0;
}

}  // namespace

bool task_small_usable(int64_t n, int64_t V, int64_t dm, int z_f32) {
    if (n < 1 || n > kTaskSmallMaxRows || V > kTaskSmallMaxV || dm > kTaskSmallMaxD || n * V > kTaskSmallMaxElems)
        return false;
    return (z_f32 ? small_cluster<float>() : small_cluster<__nv_bfloat16>()) > 0;
}

int launch_task_small(const void* Z, int z_f32, int64_t ldz, const int32_t* labels, int64_t n, int64_t V,
                      int32_t ignore, float lambda, float beta1, const void* H, const void* W, int64_t dm, float* q,
                      float* s_out, float* qhat, float* lse, float* cvec, float* wvec, void* hb_out, int hb_f32,
                      float hb_a, float hb_b, const StepScalarsIn& st, DevScalars* sc, cudaStream_t s) {
    if (!task_small_usable(n, V, dm, z_f32)) return BOM_ENOTSUP;
    TaskSmallArgs a;
    a.Z = Z;
    a.ldz = ldz;
    a.labels = labels;
    a.n = n;
    a.V = V;
    a.ignore = ignore;
    a.lambda = lambda;
    a.beta1 = beta1;
    a.H = H;
    a.W = W;
    a.dm = dm;
    a.q = q;
    a.s_out = s_out;
    a.qhat = qhat;
    a.lse = lse;
    a.cvec = cvec;
    a.wvec = wvec;
    a.hb_out = hb_out;
    a.hb_f32 = hb_f32;
    a.hb_a = hb_a;
    a.hb_b = hb_b;
    a.st = st;
    a.sc = sc;
    if (tiny_fits(n, V, dm)) {   // one CTA from shared memory
        const size_t smem = task_tiny_smem(n, V, dm);
        const cudaError_t e = z_f32 ? launch_k(task_tiny_kernel<float>, dim3(1), dim3(kSmallThreads), smem, s, a)
                                    : launch_k(task_tiny_kernel<__nv_bfloat16>, dim3(1), dim3(kSmallThreads), smem, s, a);
        if (e != cudaSuccess) return BOM_ECUDA;
        count_launch();
        return BOM_OK;
    }
    // the larger cluster only where its CTAs get work: passes of a few dozen
    // rows keep 8, whose cluster barriers cost less
    const int cmax = z_f32 ? small_cluster<float>() : small_cluster<__nv_bfloat16>();
    const int C = (n > 64 || V * dm > 65536) ? cmax : kSmallClusterMin;
    const size_t smem = task_small_smem(n, V, dm, C);
    cudaLaunchAttribute at[2];
    const cudaLaunchConfig_t cfg = small_cfg(at, C, smem, s);
    cudaError_t e;
    if (z_f32)
        e = C == kSmallClusterMax ? cudaLaunchKernelEx(&cfg, task_small_kernel<float, kSmallClusterMax>, a)
                                  : cudaLaunchKernelEx(&cfg, task_small_kernel<float, kSmallClusterMin>, a);
    else
        e = C == kSmallClusterMax ? cudaLaunchKernelEx(&cfg, task_small_kernel<__nv_bfloat16, kSmallClusterMax>, a)
                                  : cudaLaunchKernelEx(&cfg, task_small_kernel<__nv_bfloat16, kSmallClusterMin>, a);
    if (e != cudaSuccess) return BOM_ECUDA;
    count_launch();
    return BOM_OK;
}

}  // namespace bom
