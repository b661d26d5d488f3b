// RMSNorm layer of the language-model setting (the norm tensors of the
// paper's Qwen3 models, trained with weight decay 0):
//   forward   r_i = 1 / sqrt(mean_j x_ij^2 + 1e-6),  y_ij = x_ij r_i gamma_j
//   backward  dxhat = dy * gamma,
//             dx_ij = r_i (dxhat_ij - xhat_ij mean_j(dxhat_ij xhat_ij)),
//             dgamma_j = sum_i r_i dy_ij x_ij  (a weighted column sum).
// One warp per row; row sums go lane-strided in fp32 and through a fixed
// shuffle tree, so every result is deterministic.  r_i is saved for the
// backward.  HBM-bound: forward reads x and writes y, backward reads dy, x and
// writes dx (the dgamma reduction reads dy and x once more).
#include "kernels.h"

namespace bom {
namespace {

constexpr float kRmsEps = 1e-6f;

__device__ __forceinline__ float warp_sum_n(float v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    return v;
}

// Eight consecutive elements (one 16-byte word of bf16, two of fp32).
template <typename T>
__device__ __forceinline__ void load8(const T* p, float (&v)[8]) {
    if constexpr (sizeof(T) == 2) {
        const uint4 w = *reinterpret_cast<const uint4*>(p);
        const uint32_t ws[4] = {w.x, w.y, w.z, w.w};
#pragma unroll
        for (int k = 0; k < 4; ++k) {
            v[2 * k] = bf16_lo(ws[k]);
            v[2 * k + 1] = bf16_hi(ws[k]);
        }
    } else {
        const float4 a = *reinterpret_cast<const float4*>(p);
        const float4 b = *reinterpret_cast<const float4*>(p + 4);
        v[0] = a.x; v[1] = a.y; v[2] = a.z; v[3] = a.w;
        v[4] = b.x; v[5] = b.y; v[6] = b.z; v[7] = b.w;
    }
}
template <typename T>
__device__ __forceinline__ void store8(T* p, const float (&v)[8]) {
    if constexpr (sizeof(T) == 2) {
        *reinterpret_cast<uint4*>(p) = make_uint4(cvt_bf16x2(v[0], v[1]), cvt_bf16x2(v[2], v[3]),
                                                  cvt_bf16x2(v[4], v[5]), cvt_bf16x2(v[6], v[7]));
    } else {
        *reinterpret_cast<float4*>(p) = make_float4(v[0], v[1], v[2], v[3]);
        *reinterpret_cast<float4*>(p + 4) = make_float4(v[4], v[5], v[6], v[7]);
    }
}

// VEC8: rows of d % 8 == 0 elements on 16-byte aligned pitches; otherwise one
// element per lane step.
template <typename T, bool VEC8>
__global__ void __launch_bounds__(256) rmsnorm_fwd_kernel(const T* __restrict__ x, const T* __restrict__ gamma,
                                                          T* __restrict__ y, float* __restrict__ rstd, int64_t n,
                                                          int64_t d, const DevScalars* sc) {
    pdl_enter();
    if (sc->status != 0) return;
    const int64_t row = (static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x) >> 5;
    const int l = threadIdx.x & 31;
    if (row >= n) return;
    const T* xr = x + row * d;
    T* yr = y + row * d;
    float ss = 0.0f;
    if constexpr (VEC8) {
        for (int64_t j = 8 * l; j < d; j += 256) {
            float v[8];
            load8(xr + j, v);
#pragma unroll
            for (int k = 0; k < 8; ++k) ss = fmaf(v[k], v[k], ss);
        }
    } else {
        for (int64_t j = l; j < d; j += 32) {
            const float v = ld_elem(xr, j, sizeof(T) == 4);
            ss = fmaf(v, v, ss);
        }
    }
    ss = warp_sum_n(ss);
    const float r = 1.0f / sqrtf(ss / static_cast<float>(d) + kRmsEps);
    if (l == 0) rstd[row] = r;
    if constexpr (VEC8) {
        for (int64_t j = 8 * l; j < d; j += 256) {
            float v[8], g[8];
            load8(xr + j, v);
            load8(gamma + j, g);
#pragma unroll
            for (int k = 0; k < 8; ++k) v[k] = (v[k] * r) * g[k];
            store8(yr + j, v);
        }
    } else {
        for (int64_t j = l; j < d; j += 32)
            st_elem(yr, j, sizeof(T) == 4, (ld_elem(xr, j, sizeof(T) == 4) * r) * ld_elem(gamma, j, sizeof(T) == 4));
    }
}

// dx of the norm; when `pre` is given (the previous layer is Linear+GELU),
// dx is multiplied by GELU'(pre) so that it is that layer's pre-activation
// cotangent.
template <typename T, bool VEC8>
__global__ void __launch_bounds__(256) rmsnorm_bwd_kernel(const T* __restrict__ dy, const T* __restrict__ x,
                                                          const T* __restrict__ gamma, const float* __restrict__ rstd,
                                                          const T* __restrict__ pre, T* __restrict__ dx, int64_t n,
                                                          int64_t d, const DevScalars* sc) {
    pdl_enter();
    if (sc->status != 0) return;
    const int64_t row = (static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x) >> 5;
    const int l = threadIdx.x & 31;
    if (row >= n) return;
    const T* dyr = dy + row * d;
    const T* xr = x + row * d;
    T* dxr = dx + row * d;
    const float r = rstd[row];
    float dot = 0.0f;   // sum_j dxhat_j xhat_j
    if constexpr (VEC8) {
        for (int64_t j = 8 * l; j < d; j += 256) {
            float a[8], b[8], g[8];
            load8(dyr + j, a);
            load8(xr + j, b);
            load8(gamma + j, g);
#pragma unroll
            for (int k = 0; k < 8; ++k) dot = fmaf(a[k] * g[k], b[k] * r, dot);
        }
    } else {
        for (int64_t j = l; j < d; j += 32)
            dot = fmaf(ld_elem(dyr, j, sizeof(T) == 4) * ld_elem(gamma, j, sizeof(T) == 4),
                       ld_elem(xr, j, sizeof(T) == 4) * r, dot);
    }
    const float m = warp_sum_n(dot) / static_cast<float>(d);
    if constexpr (VEC8) {
        for (int64_t j = 8 * l; j < d; j += 256) {
            float a[8], b[8], g[8];
            load8(dyr + j, a);
            load8(xr + j, b);
            load8(gamma + j, g);
#pragma unroll
            for (int k = 0; k < 8; ++k) a[k] = r * (a[k] * g[k] - (b[k] * r) * m);
            if (pre) {
                float p[8];
                load8(pre + row * d + j, p);
#pragma unroll
                for (int k = 0; k < 8; ++k) a[k] *= gelu_grad_f(p[k]);
            }
            store8(dxr + j, a);
        }
    } else {
        for (int64_t j = l; j < d; j += 32) {
            float v = r * (ld_elem(dyr, j, sizeof(T) == 4) * ld_elem(gamma, j, sizeof(T) == 4) -
                           (ld_elem(xr, j, sizeof(T) == 4) * r) * m);
            if (pre) v *= gelu_grad_f(ld_elem(pre, row * d + j, sizeof(T) == 4));
            st_elem(dxr, j, sizeof(T) == 4, v);
        }
    }
}

inline unsigned cdiv_u(int64_t a, int64_t b) { return static_cast<unsigned>((a + b - 1) / b); }

}  // namespace

void launch_rmsnorm_fwd(const void* x, const void* gamma, void* y, float* rstd, int64_t n, int64_t d, int f32,
                        const DevScalars* sc, cudaStream_t s) {
    const unsigned grid = cdiv_u(n * 32, 256);
    const bool v8 = (d % 8) == 0;
    if (f32) {
        auto X = static_cast<const float*>(x);
        auto G = static_cast<const float*>(gamma);
        auto Y = static_cast<float*>(y);
        if (v8) launch_k(rmsnorm_fwd_kernel<float, true>, dim3(grid), dim3(256), 0, s, X, G, Y, rstd, n, d, sc);
        else launch_k(rmsnorm_fwd_kernel<float, false>, dim3(grid), dim3(256), 0, s, X, G, Y, rstd, n, d, sc);
    } else {
        auto X = static_cast<const __nv_bfloat16*>(x);
        auto G = static_cast<const __nv_bfloat16*>(gamma);
        auto Y = static_cast<__nv_bfloat16*>(y);
        if (v8) launch_k(rmsnorm_fwd_kernel<__nv_bfloat16, true>, dim3(grid), dim3(256), 0, s, X, G, Y, rstd, n, d, sc);
        else launch_k(rmsnorm_fwd_kernel<__nv_bfloat16, false>, dim3(grid), dim3(256), 0, s, X, G, Y, rstd, n, d, sc);
    }
    count_launch();
}

void launch_rmsnorm_bwd(const void* dy, const void* x, const void* gamma, const float* rstd, const void* pre,
                        void* dx, int64_t n, int64_t d, int f32, const DevScalars* sc, cudaStream_t s) {
    const unsigned grid = cdiv_u(n * 32, 256);
    const bool v8 = (d % 8) == 0;
    if (f32) {
        auto a = static_cast<const float*>(dy);
        auto b = static_cast<const float*>(x);
        auto g = static_cast<const float*>(gamma);
        auto p = static_cast<const float*>(pre);
        auto o = static_cast<float*>(dx);
        if (v8) launch_k(rmsnorm_bwd_kernel<float, true>, dim3(grid), dim3(256), 0, s, a, b, g, rstd, p, o, n, d, sc);
        else launch_k(rmsnorm_bwd_kernel<float, false>, dim3(grid), dim3(256), 0, s, a, b, g, rstd, p, o, n, d, sc);
    } else {
        auto a = static_cast<const __nv_bfloat16*>(dy);
        auto b = static_cast<const __nv_bfloat16*>(x);
        auto g = static_cast<const __nv_bfloat16*>(gamma);
        auto p = static_cast<const __nv_bfloat16*>(pre);
        auto o = static_cast<__nv_bfloat16*>(dx);
        if (v8) launch_k(rmsnorm_bwd_kernel<__nv_bfloat16, true>, dim3(grid), dim3(256), 0, s, a, b, g, rstd, p, o, n, d, sc);
        else launch_k(rmsnorm_bwd_kernel<__nv_bfloat16, false>, dim3(grid), dim3(256), 0, s, a, b, g, rstd, p, o, n, d, sc);
    }
    count_launch();
}

}  // namespace bom
