// Shared device-side definitions of the BOM CUDA path: the device scalar
// block of a step, the GEMM epilogue parameter block, element load/store
// helpers and the activation functions of the backbone.
#pragma once
#include <cstddef>
#include <cstdint>
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include "bom.h"

namespace bom {

// Host-side count of kernel launches made by the library (bom_launch_count).
void count_launch();

// Programmatic dependent launch.  Every kernel of the library starts with
// pdl_enter(): it lets the next kernel on the stream be scheduled (its launch
// and its prologue then overlap this kernel's tail), and waits until the
// previous kernel has completed and its memory is visible, before touching
// global memory.  Kernels launched without the attribute pass through both at
// once, so the order of the stream is kept either way.
__device__ __forceinline__ void pdl_trigger() { asm volatile("griddepcontrol.launch_dependents;" ::: "memory"); }
__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void pdl_enter() {
    pdl_trigger();
    pdl_wait();
}

// Launches kernel k with the programmatic-stream-serialization attribute.
template <typename... KArgs, typename... Args>
inline cudaError_t launch_k(void (*k)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t s,
                            Args&&... args) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = grid;
    cfg.blockDim = block;
    cfg.dynamicSmemBytes = smem;
    cfg.stream = s;
    cudaLaunchAttribute at[1];
    at[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    at[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = at;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, k, static_cast<KArgs>(args)...);
}

// Per-step scalars that live on the device so that no host round trip is
// needed between the label scan and the kernels that scale by 1/N_t.
struct DevScalars {
    int32_t status;        // latched bom_status (first error wins), 0 = OK
    int32_t n_t;           // |I_t|
    float inv_nt;          // 1 / N_t
    float coef_r[4];       // coefficient of r_i in the logit cotangent: [U, G, H, own-step pass]
    float coef_q[4];       // coefficient of the broadcast task-space vector (qhat; s_t in the own-step pass)
    float loss;            // mean CE over I_t
    float s_norm;          // ||s_t||
    float r_norm_mean;     // N_t^-1 sum_{i in I_t} ||r_i|| (own-step telemetry steps only, else 0)
    // Step scalars, written by the label scan (the first kernel of a step) from
    // host values or from the handle's device step counter, and read by the
    // kernels that need them, so a captured step replays with the current t.
    float lr;              // learning rate of the fused update
    float inv_bc1;         // 1 / (1 - beta1^t)
    float inv_bc2;         // 1 / (1 - beta2^t)
    // Row-sharded steps (bom_step_shard_begin / _end): this shard's share of
    // the supervised rows, N_t^shard / N_t, which scales its share of the
    // broadcast qhat term of the head bias gradient.
    float shard_frac;
};
// Bytes of DevScalars that bom_get_stats copies to the host (the step scalars stay).
constexpr size_t kStatsBytes = offsetof(DevScalars, lr);

// 1 / (1 - beta^t) for t >= 1, with beta^t by binary powering in double.  The
// host and the device evaluate the same correctly rounded operations in the
// same order (no contraction), so a step that takes t from the device counter
// gets the same float as one given t by the host.
__host__ __device__ inline float inv_bias_correction(float beta, int64_t t) {
    double p = 1.0, b = static_cast<double>(beta);
#ifdef __CUDA_ARCH__
    for (int64_t k = t; k > 0; k >>= 1) {
        if (k & 1) p = __dmul_rn(p, b);
        b = __dmul_rn(b, b);
    }
    return __double2float_rn(__ddiv_rn(1.0, __dsub_rn(1.0, p)));
#else
    for (int64_t k = t; k > 0; k >>= 1) {
        if (k & 1) p = p * b;
        b = b * b;
    }
    volatile double pv = p;   // keeps 1 - p a separate rounding
    return static_cast<float>(1.0 / (1.0 - pv));
#endif
}

// Weight-decay factor 1 - lr * wd, formed the same way by every update kernel.
__device__ __forceinline__ float decay_factor(float lr, float wd) { return __fmaf_rn(-lr, wd, 1.0f); }

// theta' = decay * theta - lr * q, written out so that every update kernel
// rounds the same way whatever the compiler would contract: the decayed weight
// stays exact inside one fma, only the step lr * q is rounded first.
__device__ __forceinline__ float apply_step(float decay, float th, float lr, float q) {
    return __fmaf_rn(decay, th, -__fmul_rn(lr, q));
}

__device__ __forceinline__ void latch_status(DevScalars* sc, int code) {
    atomicCAS(&sc->status, 0, code);
}

enum EpiKind : int { EPI_LINEAR = 0, EPI_LOGITS = 1, EPI_SWIGLU_FWD = 2, EPI_SWIGLU_BWD = 3, EPI_UPDATE = 4 };
enum ActKind : int { ACT_NONE = 0, ACT_GELU = 1, ACT_DGELU = 2 };

// What a GEMM does with its fp32 accumulator acc[m][n] (m: output row, n: column):
//   EPI_LINEAR     v = alpha*acc + bias[n] + beta*r1u[m]*r1v[n] + beta*mask(m)*bw[n] + resid[m][n]
//                  then ACT_GELU (out2 <- v, out <- GELU(v)), ACT_DGELU (out <- v*GELU'(aux[m][n]))
//                  or ACT_NONE (out <- v).
//   EPI_LOGITS     out <- z = acc + bias[n] rounded to the compute dtype; per (row, column tile)
//                  the pair (max_n z, sum_n exp(z - max)) goes to stats.
//   EPI_SWIGLU_FWD the accumulator tile holds [g | u] halves: out2 <- g, out3 <- u, out <- SiLU(g)*u.
//   EPI_SWIGLU_BWD acc = dA: out <- dA*u*SiLU'(g) (= dG), out2 <- dA*SiLU(g) (= dU), g = aux, u = aux2.
//   EPI_UPDATE     u = alpha*acc + beta*r1u[m]*r1v[n] is the numerator of a weight: the fused
//                  BOM-AdamW update of upd_theta / upd_v, out <- the updated weight (compute dtype).
struct EpiParams {
    float alpha_const;
    const float* alpha_dev;      // optional device factor of alpha
    float beta_const;
    const float* beta_dev;       // optional device factor of beta
    const void* bias;            // [N] compute dtype, or null
    const float* r1u;            // [M] rank-1 row factor, or null
    const float* r1v;            // [N] rank-1 column factor
    const float* bw;             // [N] broadcast-row vector, or null
    const int32_t* mask_labels;  // labels: mask(m) = labels[m] != ignore_index (null: mask = 1)
    int32_t ignore_index;
    const void* resid;           // [M, ld_resid] compute dtype, or null
    int64_t ld_resid;
    int32_t act;                 // ActKind
    int32_t in_f32;              // compute dtype of bias / resid / aux: 1 = fp32, 0 = bf16
    const void* aux;             // DGELU: pre-activation; SWIGLU_BWD: g
    int64_t ld_aux;
    const void* aux2;            // SWIGLU_BWD: u
    int64_t ld_aux2;
    void* out;
    int64_t ld_out;
    int32_t out_f32;             // dtype of out: 1 = fp32, 0 = bf16
    int32_t out2_f32;            // dtype of out2 / out3
    void* out2;
    int64_t ld_out2;
    void* out3;
    int64_t ld_out3;
    float* stats;                // EPI_LOGITS: [M, ld_stats] float2 pairs
    int64_t ld_stats;            // pairs per row (number of column tiles)
    const DevScalars* sc;        // kernels return early when sc->status != 0
    // Fused BOM-AdamW update (EPI_UPDATE; EPI_LINEAR on the SIMT and split-K
    // paths): when upd_theta is set, the epilogue value is u of the output
    // element; the epilogue advances v and theta ([M, ld_out] fp32, the
    // layout of out) and stores the updated theta into out in out's dtype
    // (the compute copy) instead of u.
    // The learning rate and 1/(1 - beta2^t) come from the step scalars in sc.
    float* upd_theta;
    float* upd_v;
    float upd_wd, upd_beta2, upd_1mb2, upd_eps;
    // Column sums of the stored output (EPI_LINEAR on the tcgen05 engine, no
    // split-K): colsum[b * ld_colsum + n] = sum of out[m, n] over the 32 rows
    // m of block b (rows past M count 0), as stored (bf16-rounded when out is
    // bf16).  Null: none.
    float* colsum;
    int64_t ld_colsum;
};

// One element of the fused update (Section 3.4): returns the new theta.
__device__ __forceinline__ float fused_update1(const EpiParams& e, int64_t idx, float u) {
    const float lr = e.sc->lr, inv_bc2 = e.sc->inv_bc2;
    float vv = e.upd_v[idx];
    float th = e.upd_theta[idx];
    vv = fmaf(e.upd_beta2, vv, e.upd_1mb2 * u * u);
    th = apply_step(decay_factor(lr, e.upd_wd), th, lr, u / (sqrtf(vv * inv_bc2) + e.upd_eps));
    e.upd_v[idx] = vv;
    e.upd_theta[idx] = th;
    return th;
}

// ------------------------------------------------------------ activations
__device__ __forceinline__ float gelu_f(float x) {
    return 0.5f * x * (1.0f + erff(x * 0.70710678118654752f));
}
__device__ __forceinline__ float gelu_grad_f(float x) {
    const float Phi = 0.5f * (1.0f + erff(x * 0.70710678118654752f));
    const float phi = 0.39894228040143268f * expf(-0.5f * x * x);
    return Phi + x * phi;
}
__device__ __forceinline__ float sigmoid_f(float x) { return 1.0f / (1.0f + expf(-x)); }
__device__ __forceinline__ float silu_f(float x) { return x * sigmoid_f(x); }
__device__ __forceinline__ float silu_grad_f(float x) {
    const float sg = sigmoid_f(x);
    return sg * (1.0f + x * (1.0f - sg));
}

// ------------------------------------------------------------ element access
__device__ __forceinline__ float ld_elem(const void* base, int64_t idx, int is_f32) {
    if (is_f32) return static_cast<const float*>(base)[idx];
    return __bfloat162float(static_cast<const __nv_bfloat16*>(base)[idx]);
}
__device__ __forceinline__ void st_elem(void* base, int64_t idx, int is_f32, float v) {
    if (is_f32)
        static_cast<float*>(base)[idx] = v;
    else
        static_cast<__nv_bfloat16*>(base)[idx] = __float2bfloat16_rn(v);
}
__device__ __forceinline__ float round_bf16(float v) { return __bfloat162float(__float2bfloat16_rn(v)); }

// Column sums of a warp's 32 x 32 block (x: this lane's row): a butterfly
// that halves the columns each lane holds at every level, so lane i returns
// the sum of column i over the 32 lanes (a fixed order, 31 shuffles).
__device__ __forceinline__ float warp_colsum32(float (&x)[32], int lane) {
#pragma unroll
    for (int s = 16; s >= 1; s >>= 1) {
        const bool up = (lane & s) != 0;
#pragma unroll
        for (int i = 0; i < s; ++i) {
            const float send = up ? x[i] : x[i + s];
            const float keep = up ? x[i + s] : x[i];
            x[i] = keep + __shfl_xor_sync(0xffffffffu, send, s);
        }
    }
    return x[0];
}

// ---------------------------------------------------------------- packed arithmetic
// Instruction-lean forms for the epilogues and streaming passes that are
// issue-bound: one instruction covers two values (sm_100 family).
constexpr float kLog2e = 1.4426950408889634f;

// Hardware base-2 exponential (PTX ex2.approx.ftz.f32: relative error about
// 2^-22; -inf gives +0).
__device__ __forceinline__ float ex2_fast(float x) {
    float y;
    asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}
// Two fp32 values rounded to nearest bf16, `lo` in the low half.
__device__ __forceinline__ uint32_t cvt_bf16x2(float lo, float hi) {
    uint32_t r;
    asm("cvt.rn.bf16x2.f32 %0, %1, %2;" : "=r"(r) : "f"(hi), "f"(lo));
    return r;
}
__device__ __forceinline__ uint32_t max_bf16x2(uint32_t a, uint32_t b) {
    uint32_t r;
    asm("max.bf16x2 %0, %1, %2;" : "=r"(r) : "r"(a), "r"(b));
    return r;
}
__device__ __forceinline__ float bf16_lo(uint32_t w) { return __uint_as_float(w << 16); }
__device__ __forceinline__ float bf16_hi(uint32_t w) { return __uint_as_float(w & 0xFFFF0000u); }
// a * b + c and a + b on fp32 pairs (fma.rn.f32x2 / add.rn.f32x2).
__device__ __forceinline__ float2 fma2(float2 a, float2 b, float2 c) {
    float2 d;
    asm("{\n\t.reg .b64 ra, rb, rc, rd;\n\t"
        "mov.b64 ra, {%2, %3};\n\tmov.b64 rb, {%4, %5};\n\tmov.b64 rc, {%6, %7};\n\t"
        "fma.rn.f32x2 rd, ra, rb, rc;\n\tmov.b64 {%0, %1}, rd;\n\t}"
        : "=f"(d.x), "=f"(d.y)
        : "f"(a.x), "f"(a.y), "f"(b.x), "f"(b.y), "f"(c.x), "f"(c.y));
    return d;
}
// Hardware square root (PTX sqrt.approx.ftz.f32).
__device__ __forceinline__ float sqrt_fast(float x) {
    float y;
    asm("sqrt.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}
// Hardware reciprocal (PTX rcp.approx.ftz.f32, about 1 ulp).
__device__ __forceinline__ float rcp_fast(float x) {
    float y;
    asm("rcp.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}
__device__ __forceinline__ float2 mul2(float2 a, float2 b) {
    float2 d;
    asm("{\n\t.reg .b64 ra, rb, rd;\n\t"
        "mov.b64 ra, {%2, %3};\n\tmov.b64 rb, {%4, %5};\n\t"
        "mul.rn.f32x2 rd, ra, rb;\n\tmov.b64 {%0, %1}, rd;\n\t}"
        : "=f"(d.x), "=f"(d.y)
        : "f"(a.x), "f"(a.y), "f"(b.x), "f"(b.y));
    return d;
}
__device__ __forceinline__ float2 add2(float2 a, float2 b) {
    float2 d;
    asm("{\n\t.reg .b64 ra, rb, rd;\n\t"
        "mov.b64 ra, {%2, %3};\n\tmov.b64 rb, {%4, %5};\n\t"
        "add.rn.f32x2 rd, ra, rb;\n\tmov.b64 {%0, %1}, rd;\n\t}"
        : "=f"(d.x), "=f"(d.y)
        : "f"(a.x), "f"(a.y), "f"(b.x), "f"(b.y));
    return d;
}
// sigma(x) = 1 / (1 + 2^(-x log2 e)) for a pair, from the two hardware
// approximations (relative error a few 1e-7: far below the bf16 outputs).
__device__ __forceinline__ float2 sigmoid2(float2 x) {
    const float2 t = mul2(x, make_float2(-kLog2e, -kLog2e));
    const float2 d = add2(make_float2(ex2_fast(t.x), ex2_fast(t.y)), make_float2(1.0f, 1.0f));
    return make_float2(rcp_fast(d.x), rcp_fast(d.y));
}

// 32 consecutive elements of one row, [n, n+32) clipped to n < N.
__device__ __forceinline__ void load_row32(const void* base, int64_t row_off, int n, int N, int is_f32,
                                           float (&v)[32]) {
    if (n + 32 <= N) {
        if (is_f32) {
            const float4* p = reinterpret_cast<const float4*>(static_cast<const float*>(base) + row_off + n);
#pragma unroll
            for (int i = 0; i < 8; ++i) {
                float4 f = p[i];
                v[4 * i] = f.x; v[4 * i + 1] = f.y; v[4 * i + 2] = f.z; v[4 * i + 3] = f.w;
            }
        } else {
            const uint4* p = reinterpret_cast<const uint4*>(static_cast<const __nv_bfloat16*>(base) + row_off + n);
#pragma unroll
            for (int i = 0; i < 4; ++i) {
                uint4 w = p[i];
                const uint32_t ws[4] = {w.x, w.y, w.z, w.w};
#pragma unroll
                for (int j = 0; j < 4; ++j) {
                    v[8 * i + 2 * j] = __uint_as_float(ws[j] << 16);
                    v[8 * i + 2 * j + 1] = __uint_as_float(ws[j] & 0xFFFF0000u);
                }
            }
        }
    } else {
#pragma unroll
        for (int i = 0; i < 32; ++i) v[i] = (n + i < N) ? ld_elem(base, row_off + n + i, is_f32) : 0.0f;
    }
}

__device__ __forceinline__ uint32_t pack_bf16x2(float lo, float hi) {
    __nv_bfloat162 h = __floats2bfloat162_rn(lo, hi);
    return *reinterpret_cast<uint32_t*>(&h);
}

// 32 bytes to a 32-byte aligned global address in one 256-bit store.
__device__ __forceinline__ void st_global_v8(void* p, uint32_t a0, uint32_t a1, uint32_t a2, uint32_t a3, uint32_t a4,
                                             uint32_t a5, uint32_t a6, uint32_t a7) {
    asm volatile("st.global.v8.b32 [%0], {%1, %2, %3, %4, %5, %6, %7, %8};" ::"l"(p), "r"(a0), "r"(a1), "r"(a2),
                 "r"(a3), "r"(a4), "r"(a5), "r"(a6), "r"(a7)
                 : "memory");
}

// One lane writes 32 values of its row.  A full chunk at a 32-byte aligned
// address leaves in 256-bit stores: each covers a whole 32-byte sector, so a
// row-per-lane store instruction makes half as many sector writes.
__device__ __forceinline__ void store_row32(void* base, int64_t row_off, int n, int N, int is_f32,
                                            const float (&v)[32]) {
    if (n + 32 <= N) {
        char* q = static_cast<char*>(base) + (row_off + n) * (is_f32 ? 4 : 2);
        if ((reinterpret_cast<uintptr_t>(q) & 31u) == 0) {
            if (is_f32) {
#pragma unroll
                for (int i = 0; i < 4; ++i)
                    st_global_v8(q + 32 * i, __float_as_uint(v[8 * i]), __float_as_uint(v[8 * i + 1]),
                                 __float_as_uint(v[8 * i + 2]), __float_as_uint(v[8 * i + 3]),
                                 __float_as_uint(v[8 * i + 4]), __float_as_uint(v[8 * i + 5]),
                                 __float_as_uint(v[8 * i + 6]), __float_as_uint(v[8 * i + 7]));
            } else {
#pragma unroll
                for (int i = 0; i < 2; ++i)
                    st_global_v8(q + 32 * i, pack_bf16x2(v[16 * i], v[16 * i + 1]),
                                 pack_bf16x2(v[16 * i + 2], v[16 * i + 3]), pack_bf16x2(v[16 * i + 4], v[16 * i + 5]),
                                 pack_bf16x2(v[16 * i + 6], v[16 * i + 7]), pack_bf16x2(v[16 * i + 8], v[16 * i + 9]),
                                 pack_bf16x2(v[16 * i + 10], v[16 * i + 11]),
                                 pack_bf16x2(v[16 * i + 12], v[16 * i + 13]),
                                 pack_bf16x2(v[16 * i + 14], v[16 * i + 15]));
            }
            return;
        }
        if (is_f32) {
            float4* p = reinterpret_cast<float4*>(static_cast<float*>(base) + row_off + n);
#pragma unroll
            for (int i = 0; i < 8; ++i) p[i] = make_float4(v[4 * i], v[4 * i + 1], v[4 * i + 2], v[4 * i + 3]);
        } else {
            uint4* p = reinterpret_cast<uint4*>(static_cast<__nv_bfloat16*>(base) + row_off + n);
#pragma unroll
            for (int i = 0; i < 4; ++i)
                p[i] = make_uint4(pack_bf16x2(v[8 * i], v[8 * i + 1]), pack_bf16x2(v[8 * i + 2], v[8 * i + 3]),
                                  pack_bf16x2(v[8 * i + 4], v[8 * i + 5]), pack_bf16x2(v[8 * i + 6], v[8 * i + 7]));
        }
    } else {
#pragma unroll
        for (int i = 0; i < 32; ++i)
            if (n + i < N) st_elem(base, row_off + n + i, is_f32, v[i]);
    }
}

__device__ __forceinline__ void load_vec32(const float* p, int n, int N, float (&v)[32]) {
    if (n + 32 <= N) {
        const float4* q = reinterpret_cast<const float4*>(p + n);
#pragma unroll
        for (int i = 0; i < 8; ++i) {
            float4 f = __ldg(q + i);
            v[4 * i] = f.x; v[4 * i + 1] = f.y; v[4 * i + 2] = f.z; v[4 * i + 3] = f.w;
        }
    } else {
#pragma unroll
        for (int i = 0; i < 32; ++i) v[i] = (n + i < N) ? p[n + i] : 0.0f;
    }
}

// Row-constant part of the EPI_LINEAR epilogue.
struct EpiRow {
    float alpha, beta_r1, beta_bw;
    bool valid;
};

__device__ __forceinline__ EpiRow epi_row(const EpiParams& e, int m, int M) {
    EpiRow r;
    const float a = e.alpha_const * (e.alpha_dev ? *e.alpha_dev : 1.0f);
    const float b = e.beta_const * (e.beta_dev ? *e.beta_dev : 1.0f);
    r.valid = m < M;
    r.alpha = a;
    r.beta_r1 = (e.r1u && r.valid) ? b * e.r1u[m] : 0.0f;
    float mask = 1.0f;
    if (e.mask_labels && r.valid) mask = (e.mask_labels[m] != e.ignore_index) ? 1.0f : 0.0f;
    r.beta_bw = e.bw ? b * mask : 0.0f;
    return r;
}

// Scalar form of EPI_LINEAR (SIMT GEMM).
__device__ __forceinline__ float epi_linear1(const EpiParams& e, const EpiRow& r, int m, int n, float acc) {
    float v = r.alpha * acc;
    if (e.bias) v += ld_elem(e.bias, n, e.in_f32);
    if (e.r1u) v += r.beta_r1 * e.r1v[n];
    if (e.bw) v += r.beta_bw * e.bw[n];
    if (e.resid) v += ld_elem(e.resid, static_cast<int64_t>(m) * e.ld_resid + n, e.in_f32);
    if (e.act == ACT_GELU) {
        st_elem(e.out2, static_cast<int64_t>(m) * e.ld_out2 + n, e.out2_f32, v);
        if (!e.out2_f32) v = round_bf16(v);
        v = gelu_f(v);
    } else if (e.act == ACT_DGELU) {
        v *= gelu_grad_f(ld_elem(e.aux, static_cast<int64_t>(m) * e.ld_aux + n, e.in_f32));
    }
    return v;
}

}  // namespace bom
