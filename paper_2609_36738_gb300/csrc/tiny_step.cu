// Whole BOM step of a small fp32 MLP classifier in one CTA.
//
// The classification settings' smallest configuration (a batch of a few dozen
// examples, widths of a few hundred, a few classes) does a million flops per
// step.  As a sequence of GEMM, task-space and update launches its step time
// is launch and pipeline latency.  Here one CTA of 1024 threads runs all of
// Algorithm 1 from shared memory after one round of global loads:
//   forward   pre_l = x_l W_l^T + b_l, x_{l+1} = GELU(pre_l) or pre_l, logits
//             z = x_L W^T + b;
//   task      label check and N_t, row log-sum-exp and CE, r_i = softmax(z_i)
//             - onehot(y_i) on I_t (0 elsewhere), s_t = N_t^-1 sum_i r_i,
//             q_t = beta1 q_{t-1} + (1-beta1) s_t, qhat_t = q_t / (1-beta1^t)
//             (Section 3.2);
//   backward  the logit cotangent N_t^-1 [(1-lambda) r_i + lambda qhat_t] on
//             I_t (Eq. mix-objective), then u of every tensor through the head
//             and the layers (Eq. mix-gradient; GELU' = Phi(x) + x phi(x));
//   update    v, theta and the compute copy of every tensor (Section 3.4), or
//             u to the caller's buffers.
// Every sum runs in a fixed order (rows, then columns, ascending), so steps are
// deterministic.  A device error (bad label, N_t = 0, a device step counter
// below 1, a non-finite row) is latched before q or any parameter is written,
// in the precedence of the multi-kernel path.
#include <atomic>

#include "kernels.h"

namespace bom {

namespace {

constexpr int kTinyThreads = 1024;
constexpr int kTinyWarps = kTinyThreads / 32;

// Row pitch of the shared-memory copies: a multiple of 4 floats (rows load as
// 16-byte words) that is 4 more than a multiple of 8, so the 16-byte words
// that eight lanes load from eight consecutive rows at one column fall in
// different bank quads; the padding columns stay zero.
__host__ __device__ inline int tiny_pitch(int d) { return ((d + 7) & ~7) + 4; }

__device__ __forceinline__ float tw_sum(float v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    return v;
}
__device__ __forceinline__ float tw_max(float v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
    return v;
}

// Fills dst[r * pitch + c] = src[r * cols + c] for r < rows, c < cols.
__device__ __forceinline__ void tiny_stage(float* dst, const float* src, int rows, int cols, int pitch) {
    for (int i = threadIdx.x; i < rows * cols; i += kTinyThreads) {
        const int r = i / cols, c = i - r * cols;
        dst[r * pitch + c] = src[i];
    }
}

__global__ void __launch_bounds__(kTinyThreads, 1) tiny_step_kernel(const TinyStepArgs a) {
    pdl_enter();
    extern __shared__ float sm[];
    __shared__ float wf[kTinyWarps];
    __shared__ int wi[3][kTinyWarps];
    __shared__ int s_code;
    __shared__ float s_inv, s_bc1, s_bc2, s_lr;
    const int tid = threadIdx.x, w = tid >> 5, l = tid & 31;
    const int n = a.n, nl = a.nl, V = a.dim[nl + 1];
    const TinyLayout& L = a.lay;
    if (a.sc->status != 0) return;   // an earlier kernel of the step failed

    // ---------------------------------------------------------------- loads
    for (int i = tid; i < L.floats; i += kTinyThreads) sm[i] = 0.0f;   // zero padding
    __syncthreads();
    tiny_stage(sm + L.x, a.x, n, a.dim[0], tiny_pitch(a.dim[0]));
    for (int k = 0; k <= nl; ++k) {
        tiny_stage(sm + L.W[k], a.W[k], a.dim[k + 1], a.dim[k], tiny_pitch(a.dim[k]));
        if (a.b[k] != nullptr)
            for (int j = tid; j < a.dim[k + 1]; j += kTinyThreads) sm[L.b[k] + j] = a.b[k][j];
    }
    int* lab = reinterpret_cast<int*>(sm + L.lab);
    for (int i = tid; i < n; i += kTinyThreads) lab[i] = a.labels[i];
    if (tid == 0) {
        int64_t t = 1;
        if (a.st.t_dev != nullptr) t = __ldcg(a.st.t_dev);
        s_lr = a.st.lr_dev != nullptr ? __ldcg(a.st.lr_dev) : a.st.lr;
        s_bc1 = a.st.t_dev != nullptr ? (t >= 1 ? inv_bias_correction(a.st.beta1, t) : 0.0f) : a.st.inv_bc1;
        s_bc2 = a.st.t_dev != nullptr ? (t >= 1 ? inv_bias_correction(a.st.beta2, t) : 0.0f) : a.st.inv_bc2;
        s_code = (a.st.t_dev != nullptr && t < 1) ? BOM_EINVAL : 0;
    }
    __syncthreads();

    // ---------------------------------------------------------------- forward
    // act(k) is the input of layer k (the head for k = nl)
    auto act = [&](int k) -> float* { return k == 0 ? sm + L.x : sm + L.act[k - 1]; };
    for (int k = 0; k <= nl; ++k) {
        const int din = a.dim[k], dout = a.dim[k + 1], pin = tiny_pitch(din), pout = tiny_pitch(dout);
        const float* xin = act(k);
        const float* W = sm + L.W[k];
        const float* b = a.b[k] != nullptr ? sm + L.b[k] : nullptr;
        float* pre = k < nl ? sm + L.pre[k] : sm + L.z;
        float* out = k < nl ? sm + L.act[k] : nullptr;
        const bool gelu = k < nl && a.gelu[k];
        // four rows per thread: each 16-byte word of W serves four rows
        const int nb = (n + 3) >> 2, c4 = (din + 3) >> 2;
        for (int i0 = tid; i0 < nb * dout; i0 += kTinyThreads) {
            const int ib = i0 / dout, j = i0 - ib * dout;
            const int nr = min(4, n - 4 * ib);
            const float4* wr = reinterpret_cast<const float4*>(W + j * pin);
            float acc[4] = {0.0f, 0.0f, 0.0f, 0.0f};
            for (int c = 0; c < c4; ++c) {
                const float4 wv = wr[c];
#pragma unroll
                for (int r = 0; r < 4; ++r) {
                    if (r >= nr) break;
                    const float4 xv = reinterpret_cast<const float4*>(xin + (4 * ib + r) * pin)[c];
                    acc[r] = fmaf(xv.x, wv.x, acc[r]);
                    acc[r] = fmaf(xv.y, wv.y, acc[r]);
                    acc[r] = fmaf(xv.z, wv.z, acc[r]);
                    acc[r] = fmaf(xv.w, wv.w, acc[r]);
                }
            }
#pragma unroll
            for (int r = 0; r < 4; ++r) {
                if (r >= nr) break;
                const int i = 4 * ib + r;
                float v = acc[r];
                if (b) v += b[j];
                pre[i * pout + j] = v;
                if (out) out[i * pout + j] = gelu ? gelu_f(v) : v;
            }
        }
        __syncthreads();
    }

    // ---------------------------------------------------------------- task space
    float* Z = sm + L.z;          // logits, then R, then the logit cotangent
    float* lse = sm + L.lse;
    const int pv = tiny_pitch(V);
    {
        float ce_w = 0.0f;
        int nt_w = 0, bad_w = 0, nf_w = 0;
        for (int r = w; r < n; r += kTinyWarps) {
            const int y = lab[r];
            const bool sup = y != a.ignore;
            const bool ok_y = sup && y >= 0 && y < V;
            const float* zr = Z + r * pv;
            float m = -INFINITY;
            for (int j = l; j < V; j += 32) m = fmaxf(m, zr[j]);
            m = tw_max(m);
            float sum = 0.0f;
            for (int j = l; j < V; j += 32) sum += expf(zr[j] - m);
            sum = tw_sum(sum);
            if (l == 0) {
                const float Lr = m + logf(sum);
                const float zy = ok_y ? zr[y] : 0.0f;
                lse[r] = Lr;
                if (sup && !ok_y) ++bad_w;
                if (ok_y) {
                    ++nt_w;
                    ce_w += Lr - zy;
                }
                if (!isfinite(Lr) || (ok_y && !isfinite(zy))) ++nf_w;
                lab[r] = ok_y ? y : -1;   // -1: not in I_t
            }
        }
        if (l == 0) {
            wf[w] = ce_w;
            wi[0][w] = nt_w;
            wi[1][w] = bad_w;
            wi[2][w] = nf_w;
        }
    }
    __syncthreads();
    if (tid == 0) {
        float ce = 0.0f;
        int nt = 0, bad = 0, nf = 0;
        for (int k = 0; k < kTinyWarps; ++k) {
            ce += wf[k];
            nt += wi[0][k];
            bad += wi[1][k];
            nf += wi[2][k];
        }
        int code = 0;
        if (bad > 0)
            code = BOM_ELABEL;
        else if (nt == 0)
            code = BOM_EEMPTY;
        else if (s_code != 0)
            code = s_code;
        else if (nf > 0)
            code = BOM_ENONFINITE;
        s_code = code;
        s_inv = nt > 0 ? 1.0f / static_cast<float>(nt) : 0.0f;
        DevScalars* sc = a.sc;
        if (code != 0) latch_status(sc, code);
        const float inv = s_inv;
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
    __syncthreads();
    if (s_code != 0) return;   // q and every parameter stay as they were

    // R over Z (0 on rows outside I_t)
    for (int i0 = tid; i0 < n * V; i0 += kTinyThreads) {
        const int r = i0 / V, j = i0 - r * V;
        const int y = lab[r];
        float p = 0.0f;
        if (y >= 0) {
            p = expf(Z[r * pv + j] - lse[r]);
            if (j == y) p -= 1.0f;
        }
        Z[r * pv + j] = p;
    }
    __syncthreads();
    // s_t, q_t, qhat_t; the row log-sum-exp out
    float* qh = sm + L.qh;
    float* sv = sm + L.sv;
    {
        const float inv = s_inv;
        float ss = 0.0f;
        for (int j = tid; j < V; j += kTinyThreads) {
            float acc = 0.0f;
            for (int r = 0; r < n; ++r) acc += Z[r * pv + j];
            const float s = acc * inv;
            const float qn = a.beta1 * a.q[j] + (1.0f - a.beta1) * s;
            const float qhat = qn * s_bc1;
            a.q[j] = qn;
            a.s_out[j] = s;
            a.qhat_out[j] = qhat;
            qh[j] = qhat;
            sv[j] = s;
            ss += s * s;
        }
        for (int r = tid; r < n; r += kTinyThreads) a.lse_out[r] = lse[r];
        ss = tw_sum(ss);
        if (l == 0) wf[w] = ss;
    }
    __syncthreads();
    if (tid == 0) {
        float t = 0.0f;
        for (int k = 0; k < kTinyWarps; ++k) t += wf[k];
        a.sc->s_norm = sqrtf(t);
    }
    // the logit cotangent N_t^-1 [(1-lambda) r_i + lambda qhat] on I_t
    {
        const float ca = (1.0f - a.lambda) * s_inv, cb = a.lambda * s_inv;
        for (int i0 = tid; i0 < n * V; i0 += kTinyThreads) {
            const int r = i0 / V, j = i0 - r * V;
            Z[r * pv + j] = lab[r] >= 0 ? fmaf(ca, Z[r * pv + j], cb * qh[j]) : 0.0f;
        }
    }
    __syncthreads();

    // ---------------------------------------------------------------- backward
    // u of a tensor: fused BOM-AdamW update of theta, v and the compute copy,
    // or u to the caller's buffer
    const float lr = s_lr, inv_bc2 = s_bc2, beta2 = a.beta2, omb2 = 1.0f - a.beta2, eps = a.eps;
    auto emit = [&](int t, int64_t idx, float u) {
        if (a.theta[t] == nullptr) {
            a.u[t][idx] = u;
            return;
        }
        float vv = a.v[t][idx];
        float th = a.theta[t][idx];
        vv = fmaf(beta2, vv, omb2 * u * u);
        th = apply_step(decay_factor(lr, a.wd[t]), th, lr, u / (sqrtf(vv * inv_bc2) + eps));
        a.v[t][idx] = vv;
        a.theta[t][idx] = th;
        a.copy[t][idx] = th;
    };
    // dcur: the cotangent of the output of layer k (pre-activation after GELU')
    float* dcur = Z;
    int pcur = pv;
    for (int k = nl; k >= 0; --k) {
        const int din = a.dim[k], dout = a.dim[k + 1], pin = tiny_pitch(din);
        const float* xin = act(k);
        const float* W = sm + L.W[k];
        const int tw = a.tw[k], tb = a.tb[k];
        // weight: u_W[j, c] = sum_i dcur[i, j] xin[i, c], four output rows j per
        // thread (one 16-byte word of dcur per row i serves all four)
        const int jb4 = (dout + 3) >> 2;
        for (int i0 = tid; i0 < jb4 * din; i0 += kTinyThreads) {
            const int jb = i0 / din, c = i0 - jb * din;
            float acc[4] = {0.0f, 0.0f, 0.0f, 0.0f};
            for (int r = 0; r < n; ++r) {
                const float4 dv = reinterpret_cast<const float4*>(dcur + r * pcur)[jb];
                const float xv = xin[r * pin + c];
                acc[0] = fmaf(dv.x, xv, acc[0]);
                acc[1] = fmaf(dv.y, xv, acc[1]);
                acc[2] = fmaf(dv.z, xv, acc[2]);
                acc[3] = fmaf(dv.w, xv, acc[3]);
            }
#pragma unroll
            for (int q = 0; q < 4; ++q)
                if (4 * jb + q < dout) emit(tw, static_cast<int64_t>(4 * jb + q) * din + c, acc[q]);
        }
        // bias: the head's is (1-lambda) s + lambda qhat, a layer's the column sum of its cotangent
        if (tb >= 0)
            for (int j = tid; j < dout; j += kTinyThreads) {
                float acc;
                if (k == nl) {
                    acc = (1.0f - a.lambda) * sv[j] + a.lambda * qh[j];
                } else {
                    acc = 0.0f;
                    for (int r = 0; r < n; ++r) acc += dcur[r * pcur + j];
                }
                emit(tb, j, acc);
            }
        if (k == 0) break;
        // input: dnext[i, c] = sum_j dcur[i, j] W[j, c], times GELU'(pre) of layer k-1
        float* dnext = sm + (dcur == sm + L.g[0] ? L.g[1] : L.g[0]);
        const float* pre = sm + L.pre[k - 1];
        const bool gelu = a.gelu[k - 1];
        for (int i0 = tid; i0 < n * din; i0 += kTinyThreads) {
            const int r = i0 / din, c = i0 - r * din;
            float acc = 0.0f;
            for (int j = 0; j < dout; ++j) acc = fmaf(dcur[r * pcur + j], W[j * pin + c], acc);
            if (gelu) acc *= gelu_grad_f(pre[r * pin + c]);
            dnext[r * pin + c] = acc;
        }
        __syncthreads();   // dnext complete; every read of dcur done
        dcur = dnext;
        pcur = pin;
    }
    if (tid == 0 && a.t_adv != nullptr) *a.t_adv += 1;   // the step latched no error
}

}  // namespace

// Shared-memory layout (in floats) of tiny_step_kernel for these dimensions,
// and whether it fits.
bool tiny_step_layout(int n, int nl, const int* dim, const bool* bias, TinyLayout* lay) {
    if (n < 1 || n > kTinyStepMaxRows || nl < 0 || nl > kTinyStepMaxLayers) return false;
    int64_t off = 0;
    auto take = [&](int64_t floats) {
        const int64_t o = off;
        off += (floats + 3) & ~int64_t(3);
        return static_cast<int>(o);
    };
    TinyLayout L{};
    for (int k = 0; k <= nl + 1; ++k)
        if (dim[k] < 1 || dim[k] > kTinyStepMaxWidth) return false;
    const int V = dim[nl + 1];
    L.x = take(int64_t(n) * tiny_pitch(dim[0]));
    int maxw = 1;
    for (int k = 0; k <= nl; ++k) {
        L.W[k] = take(int64_t(dim[k + 1]) * tiny_pitch(dim[k]));
        L.b[k] = bias[k] ? take(dim[k + 1]) : 0;
        if (k < nl) {
            L.pre[k] = take(int64_t(n) * tiny_pitch(dim[k + 1]));
            L.act[k] = take(int64_t(n) * tiny_pitch(dim[k + 1]));
            maxw = dim[k + 1] > maxw ? dim[k + 1] : maxw;
        }
    }
    L.z = take(int64_t(n) * tiny_pitch(V));
    L.g[0] = take(int64_t(n) * tiny_pitch(maxw));
    L.g[1] = take(int64_t(n) * tiny_pitch(maxw));
    L.lse = take(n);
    L.lab = take(n);
    L.qh = take(V);
    L.sv = take(V);
    L.floats = static_cast<int>(off);
    if (off > kTinyStepMaxFloats) return false;
    *lay = L;
    return true;
}

int launch_tiny_step(const TinyStepArgs& a, cudaStream_t s) {
    const size_t smem = static_cast<size_t>(a.lay.floats) * 4;
    constexpr int kMaxDev = 64;
    static std::atomic<int> ready[kMaxDev];   // the shared-memory attribute is a per-device setting
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDev) return BOM_ECUDA;
    if (ready[dev].load(std::memory_order_relaxed) == 0) {
        if (cudaFuncSetAttribute(tiny_step_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 static_cast<int>(kTinyStepMaxFloats * 4)) != cudaSuccess)
            return BOM_ECUDA;
        ready[dev].store(1, std::memory_order_relaxed);
    }
    launch_k(tiny_step_kernel, dim3(1), dim3(kTinyThreads), smem, s, a);
    count_launch();
    return cudaPeekAtLastError() == cudaSuccess ? BOM_OK : BOM_ECUDA;
}

}  // namespace bom
