// BOM-AdamW update (Section 3.4; Algorithm 1, last two steps), one HBM pass:
//   u     = g                      (numerator supplied directly), or
//   u     = (1-lambda) g + lambda h  (Eq. mix-gradient, from separate g and h)
//   v    <- beta2 v + (1-beta2) u^2
//   theta <- (1 - lr wd) theta - lr u / (sqrt(v / (1-beta2^t)) + eps)
// There is no first-moment buffer and no first-moment bias correction.
// Each thread moves 4 elements per access with 128-bit (fp32) / 64-bit (bf16)
// streaming loads and stores; the grid is a multiple of the SM count and
// strides over the range.
//
// BOM-Adam-mini (Section 3.5, composition with Adam-mini) shares one second
// moment per block of `block` consecutive elements:
//   v_b  <- beta2 v_b + (1-beta2) mean_{i in b} u_i^2
//   theta <- (1 - lr wd) theta - lr u / (sqrt(v_b / (1-beta2^t)) + eps)
// One CTA per block (grid-stride over blocks): a first sweep forms sum u^2 in
// a fixed order, thread 0 advances v_b, a second sweep applies the update; the
// second sweep's reads of g and h hit L2.
#include <atomic>
#include "kernels.h"
#include "tc_ptx.cuh"
#include <mutex>
#include <type_traits>

namespace bom {

int device_sm_count();

namespace {

struct UpdCoef {
    float lr, wd, decay, lam, beta2, one_m_beta2, eps, inv_bc2;
    int from_step;   // take lr and inv_bc2 from the step scalars (updates inside bom_step)
};

// The coefficients a kernel uses: lr and 1/(1 - beta2^t) from the step
// scalars when asked, and the decay factor formed on the device.
__device__ __forceinline__ UpdCoef resolve_coef(UpdCoef c, const DevScalars* sc) {
    if (c.from_step && sc != nullptr) {
        c.lr = sc->lr;
        c.inv_bc2 = sc->inv_bc2;
    }
    c.decay = decay_factor(c.lr, c.wd);
    return c;
}

__device__ __forceinline__ float upd1(float& th, float& vv, float u, const UpdCoef& c) {
    vv = fmaf(c.beta2, vv, c.one_m_beta2 * u * u);
    const float den = sqrtf(vv * c.inv_bc2) + c.eps;
    th = apply_step(c.decay, th, c.lr, u / den);
    return th;
}

// Factor of global-norm clipping: min(1, max_norm / (||u|| + 1e-6)).
__device__ __forceinline__ float clip_scale(const double* sq, float max_norm) {
    return static_cast<float>(fmin(1.0, static_cast<double>(max_norm) / (sqrt(*sq) + 1e-6)));
}

template <bool G_BF16, bool HAS_H, bool SHADOW, bool CLIP>
__global__ void __launch_bounds__(256) update_kernel(float* __restrict__ theta, const void* __restrict__ g,
                                                     const float* __restrict__ h, float* __restrict__ v,
                                                     uint16_t* __restrict__ shadow, int64_t n, UpdCoef c_in,
                                                     const double* __restrict__ clip_sq, float max_norm,
                                                     const DevScalars* sc) {
    pdl_enter();
    if (sc != nullptr && sc->status != 0) return;   // inside a step that latched an error
    const UpdCoef c = resolve_coef(c_in, sc);
    const float cs = CLIP ? clip_scale(clip_sq, max_norm) : 1.0f;
    const int64_t n4 = n >> 2;
    const int64_t stride = static_cast<int64_t>(gridDim.x) * blockDim.x;
    for (int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; i < n4; i += stride) {
        float4 th = __ldcs(reinterpret_cast<const float4*>(theta) + i);
        float4 vv = __ldcs(reinterpret_cast<const float4*>(v) + i);
        float u[4];
        if constexpr (G_BF16) {
            const uint2 w = __ldcs(reinterpret_cast<const uint2*>(g) + i);
            u[0] = __uint_as_float(w.x << 16);
            u[1] = __uint_as_float(w.x & 0xFFFF0000u);
            u[2] = __uint_as_float(w.y << 16);
            u[3] = __uint_as_float(w.y & 0xFFFF0000u);
        } else {
            const float4 f = __ldcs(reinterpret_cast<const float4*>(g) + i);
            u[0] = f.x; u[1] = f.y; u[2] = f.z; u[3] = f.w;
        }
        if constexpr (HAS_H) {
            const float4 hh = __ldcs(reinterpret_cast<const float4*>(h) + i);
            const float om = 1.0f - c.lam;
            u[0] = om * u[0] + c.lam * hh.x;
            u[1] = om * u[1] + c.lam * hh.y;
            u[2] = om * u[2] + c.lam * hh.z;
            u[3] = om * u[3] + c.lam * hh.w;
        }
        if constexpr (CLIP) {
#pragma unroll
            for (int k = 0; k < 4; ++k) u[k] *= cs;
        }
        upd1(th.x, vv.x, u[0], c);
        upd1(th.y, vv.y, u[1], c);
        upd1(th.z, vv.z, u[2], c);
        upd1(th.w, vv.w, u[3], c);
        __stcs(reinterpret_cast<float4*>(theta) + i, th);
        __stcs(reinterpret_cast<float4*>(v) + i, vv);
        if constexpr (SHADOW) {
            uint2 sh;
            sh.x = pack_bf16x2(th.x, th.y);
            sh.y = pack_bf16x2(th.z, th.w);
            __stcs(reinterpret_cast<uint2*>(shadow) + i, sh);
        }
    }
    // tail (n not a multiple of 4)
    const int64_t t = (n4 << 2) + static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x;
    if (t < n && t < (n4 << 2) + 4) {
        float u = G_BF16 ? __bfloat162float(static_cast<const __nv_bfloat16*>(g)[t]) : static_cast<const float*>(g)[t];
        if (HAS_H) u = (1.0f - c.lam) * u + c.lam * h[t];
        if (CLIP) u *= cs;
        float th = theta[t], vv = v[t];
        upd1(th, vv, u, c);
        theta[t] = th;
        v[t] = vv;
        if (SHADOW) reinterpret_cast<__nv_bfloat16*>(shadow)[t] = __float2bfloat16_rn(th);
    }
}

__device__ __forceinline__ float warp_sum_f(float v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    return v;
}

// u of VEC consecutive elements starting at i.
template <bool G_BF16, bool HAS_H, int VEC>
__device__ __forceinline__ void load_u(const void* g, const float* h, int64_t i, float lam, float (&u)[VEC]) {
    if constexpr (VEC == 4) {
        if constexpr (G_BF16) {
            const uint2 w = *(reinterpret_cast<const uint2*>(static_cast<const uint16_t*>(g) + i));
            u[0] = __uint_as_float(w.x << 16);
            u[1] = __uint_as_float(w.x & 0xFFFF0000u);
            u[2] = __uint_as_float(w.y << 16);
            u[3] = __uint_as_float(w.y & 0xFFFF0000u);
        } else {
            const float4 f = *(reinterpret_cast<const float4*>(static_cast<const float*>(g) + i));
            u[0] = f.x; u[1] = f.y; u[2] = f.z; u[3] = f.w;
        }
        if constexpr (HAS_H) {
            const float4 hh = *(reinterpret_cast<const float4*>(h + i));
            const float hv[4] = {hh.x, hh.y, hh.z, hh.w};
#pragma unroll
            for (int k = 0; k < 4; ++k) u[k] = (1.0f - lam) * u[k] + lam * hv[k];
        }
    } else {
#pragma unroll
        for (int k = 0; k < VEC; ++k) {
            float x = G_BF16 ? __bfloat162float(static_cast<const __nv_bfloat16*>(g)[i + k])
                             : static_cast<const float*>(g)[i + k];
            if (HAS_H) x = (1.0f - lam) * x + lam * h[i + k];
            u[k] = x;
        }
    }
}

// Blocks larger than a CTA holds in registers: a cluster of kBlockCluster
// CTAs takes one block at a time, so a few large blocks (a whole-tensor block
// of a big weight) still spread over many SMs.  Each CTA sums u^2 over its
// interleaved share of the block; after a cluster barrier the leading CTA adds
// the CTA partials from distributed shared memory in rank order (fixed order:
// deterministic), advances v_b and publishes the denominator, which every CTA
// reads back after a second barrier; then all update their share (the second
// read of u mostly hits L2: the cluster's block is its whole working set).
// Every CTA of a cluster walks the same blocks, so all meet every barrier.
constexpr int kBlockCluster = 8;

template <bool G_BF16, bool HAS_H, bool SHADOW, int VEC>
__global__ void __launch_bounds__(256) update_blockshared_cluster_kernel(float* __restrict__ theta,
                                                                         const void* __restrict__ g,
                                                                         const float* __restrict__ h,
                                                                         float* __restrict__ vb,
                                                                         uint16_t* __restrict__ shadow, int64_t n,
                                                                         int64_t block, UpdCoef c_in) {
    pdl_enter();
    __shared__ float red[8];
    __shared__ float s_part;   // this CTA's sum of u^2 over its share of the block
    __shared__ float s_den;    // leading CTA: the block's denominator
    __shared__ float s_den_local;
    const UpdCoef c = resolve_coef(c_in, nullptr);
    const uint32_t rank = cluster_ctarank();
    const int64_t ncl = gridDim.x / kBlockCluster;
    const int64_t nb = (n + block - 1) / block;
    const int64_t stride = static_cast<int64_t>(kBlockCluster) * 256 * VEC;
    for (int64_t b = blockIdx.x / kBlockCluster; b < nb; b += ncl) {
        const int64_t e0 = b * block;
        const int64_t e1 = e0 + block < n ? e0 + block : n;
        const int64_t i0 = e0 + (static_cast<int64_t>(rank) * 256 + threadIdx.x) * VEC;
        float acc = 0.0f;
        int64_t i = i0;
        for (; i + 3 * stride < e1; i += 4 * stride) {   // four loads in flight per thread
            float u[4][VEC];
#pragma unroll
            for (int j = 0; j < 4; ++j) load_u<G_BF16, HAS_H, VEC>(g, h, i + j * stride, c.lam, u[j]);
#pragma unroll
            for (int j = 0; j < 4; ++j)
#pragma unroll
                for (int k = 0; k < VEC; ++k) acc = fmaf(u[j][k], u[j][k], acc);
        }
        for (; i < e1; i += stride) {
            float u[VEC];
            load_u<G_BF16, HAS_H, VEC>(g, h, i, c.lam, u);
#pragma unroll
            for (int k = 0; k < VEC; ++k) acc = fmaf(u[k], u[k], acc);
        }
        acc = warp_sum_f(acc);
        if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = acc;
        __syncthreads();
        if (threadIdx.x == 0) {
            float tot = 0.0f;
#pragma unroll
            for (int w = 0; w < 8; ++w) tot += red[w];
            s_part = tot;
        }
        cluster_sync();   // every CTA's s_part is written
        if (rank == 0 && threadIdx.x == 0) {
            float tot = 0.0f;
            for (uint32_t r = 0; r < kBlockCluster; ++r) tot += ld_shared_cluster_f32(mapa_shared(smem_u32(&s_part), r));
            const float vv = fmaf(c.beta2, vb[b], c.one_m_beta2 * (tot / static_cast<float>(e1 - e0)));
            vb[b] = vv;
            s_den = sqrtf(vv * c.inv_bc2) + c.eps;
        }
        cluster_sync();   // s_den is written; every s_part has been read
        if (threadIdx.x == 0) s_den_local = ld_shared_cluster_f32(mapa_shared(smem_u32(&s_den), 0));
        __syncthreads();
        const float den = s_den_local;
#pragma unroll 2
        for (int64_t i = i0; i < e1; i += stride) {
            float u[VEC];
            load_u<G_BF16, HAS_H, VEC>(g, h, i, c.lam, u);
            if constexpr (VEC == 4) {
                float4 th = __ldcs(reinterpret_cast<const float4*>(theta + i));
                th.x = apply_step(c.decay, th.x, c.lr, u[0] / den);
                th.y = apply_step(c.decay, th.y, c.lr, u[1] / den);
                th.z = apply_step(c.decay, th.z, c.lr, u[2] / den);
                th.w = apply_step(c.decay, th.w, c.lr, u[3] / den);
                __stcs(reinterpret_cast<float4*>(theta + i), th);
                if constexpr (SHADOW) {
                    uint2 sh;
                    sh.x = pack_bf16x2(th.x, th.y);
                    sh.y = pack_bf16x2(th.z, th.w);
                    __stcs(reinterpret_cast<uint2*>(shadow + i), sh);
                }
            } else {
#pragma unroll
                for (int k = 0; k < VEC; ++k) {
                    const float th = apply_step(c.decay, theta[i + k], c.lr, u[k] / den);
                    theta[i + k] = th;
                    if (SHADOW) reinterpret_cast<__nv_bfloat16*>(shadow)[i + k] = __float2bfloat16_rn(th);
                }
            }
        }
        // s_den_local and red are rewritten only after the next block's first
        // cluster barrier, which every thread of this CTA reaches after its reads
    }
    cluster_sync();   // no CTA leaves while another may still read its shared memory
}

// Fewer large blocks than the GPU runs clusters at once (a whole-tensor block
// of a big weight): the whole grid works on them in three launches.
//   bs_chunk_sq   part[b * S + j] = sum of u^2 over chunk j of block b (chunks
//                 of `ch` elements, fixed order within a chunk);
//   bs_finish     one warp per block adds its S partials (lane-strided, then a
//                 fixed shuffle tree), advances v_b and writes the denominator;
//   bs_apply      the elementwise update with its block's denominator.
template <bool G_BF16, bool HAS_H, int VEC>
__global__ void __launch_bounds__(256) bs_chunk_sq_kernel(const void* __restrict__ g, const float* __restrict__ h,
                                                          float lam, int64_t n, int64_t block, int64_t ch, int64_t S,
                                                          int64_t nchunks, float* __restrict__ part) {
    pdl_enter();
    __shared__ float red[8];
    for (int64_t cidx = blockIdx.x; cidx < nchunks; cidx += gridDim.x) {
        const int64_t b = cidx / S, j = cidx - b * S;
        const int64_t e0 = b * block + j * ch;
        int64_t e1 = b * block + block < n ? b * block + block : n;
        if (e0 + ch < e1) e1 = e0 + ch;
        const int64_t st = 256 * VEC;
        float acc = 0.0f;
        int64_t i = e0 + static_cast<int64_t>(threadIdx.x) * VEC;
        for (; i + 3 * st < e1; i += 4 * st) {   // four loads in flight per thread
            float u[4][VEC];
#pragma unroll
            for (int q = 0; q < 4; ++q) load_u<G_BF16, HAS_H, VEC>(g, h, i + q * st, lam, u[q]);
#pragma unroll
            for (int q = 0; q < 4; ++q)
#pragma unroll
                for (int k = 0; k < VEC; ++k) acc = fmaf(u[q][k], u[q][k], acc);
        }
        for (; i < e1; i += st) {
            float u[VEC];
            load_u<G_BF16, HAS_H, VEC>(g, h, i, lam, u);
#pragma unroll
            for (int k = 0; k < VEC; ++k) acc = fmaf(u[k], u[k], acc);
        }
        acc = warp_sum_f(acc);
        if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = acc;
        __syncthreads();
        if (threadIdx.x == 0) {
            float tot = 0.0f;
#pragma unroll
            for (int w = 0; w < 8; ++w) tot += red[w];
            part[cidx] = tot;
        }
        __syncthreads();
    }
}

__global__ void __launch_bounds__(256) bs_finish_kernel(const float* __restrict__ part, int64_t S, int64_t nb,
                                                        int64_t n, int64_t block, float* __restrict__ vb,
                                                        float* __restrict__ den, UpdCoef c_in) {
    pdl_enter();
    const UpdCoef c = resolve_coef(c_in, nullptr);
    const int64_t b = static_cast<int64_t>(blockIdx.x) * 8 + (threadIdx.x >> 5);
    const int lane = threadIdx.x & 31;
    if (b >= nb) return;
    float t = 0.0f;
    for (int64_t j = lane; j < S; j += 32) t += part[b * S + j];
    t = warp_sum_f(t);
    if (lane == 0) {
        const int64_t len = b * block + block < n ? block : n - b * block;
        const float vv = fmaf(c.beta2, vb[b], c.one_m_beta2 * (t / static_cast<float>(len)));
        vb[b] = vv;
        den[b] = sqrtf(vv * c.inv_bc2) + c.eps;
    }
}

template <bool G_BF16, bool HAS_H, bool SHADOW, int VEC>
__global__ void __launch_bounds__(256) bs_apply_kernel(float* __restrict__ theta, const void* __restrict__ g,
                                                       const float* __restrict__ h, uint16_t* __restrict__ shadow,
                                                       int64_t n, int64_t block, const float* __restrict__ den,
                                                       UpdCoef c_in) {
    pdl_enter();
    const UpdCoef c = resolve_coef(c_in, nullptr);
    const int64_t nv = n / VEC;   // VEC = 4 only when n and block are multiples of 4
    const int64_t stride = static_cast<int64_t>(gridDim.x) * 256;
    for (int64_t q = static_cast<int64_t>(blockIdx.x) * 256 + threadIdx.x; q < nv; q += stride) {
        const int64_t i = q * VEC;
        const float d = den[i / block];   // a group of VEC elements never straddles two blocks
        float u[VEC];
        load_u<G_BF16, HAS_H, VEC>(g, h, i, c.lam, u);
        if constexpr (VEC == 4) {
            float4 th = __ldcs(reinterpret_cast<const float4*>(theta + i));
            th.x = apply_step(c.decay, th.x, c.lr, u[0] / d);
            th.y = apply_step(c.decay, th.y, c.lr, u[1] / d);
            th.z = apply_step(c.decay, th.z, c.lr, u[2] / d);
            th.w = apply_step(c.decay, th.w, c.lr, u[3] / d);
            __stcs(reinterpret_cast<float4*>(theta + i), th);
            if constexpr (SHADOW) {
                uint2 sh;
                sh.x = pack_bf16x2(th.x, th.y);
                sh.y = pack_bf16x2(th.z, th.w);
                __stcs(reinterpret_cast<uint2*>(shadow + i), sh);
            }
        } else {
            const float th = apply_step(c.decay, theta[i], c.lr, u[0] / d);
            theta[i] = th;
            if (SHADOW) reinterpret_cast<__nv_bfloat16*>(shadow)[i] = __float2bfloat16_rn(th);
        }
    }
}

template <bool G_BF16, bool HAS_H, bool SHADOW, int VEC>
__global__ void __launch_bounds__(256) update_blockshared_kernel(float* __restrict__ theta, const void* __restrict__ g,
                                                                 const float* __restrict__ h, float* __restrict__ vb,
                                                                 uint16_t* __restrict__ shadow, int64_t n,
                                                                 int64_t block, UpdCoef c_in) {
    pdl_enter();
    __shared__ float red[8];
    __shared__ float s_den;
    const UpdCoef c = resolve_coef(c_in, nullptr);
    const int64_t nb = (n + block - 1) / block;
    for (int64_t b = blockIdx.x; b < nb; b += gridDim.x) {
        const int64_t e0 = b * block;
        const int64_t e1 = e0 + block < n ? e0 + block : n;
        float acc = 0.0f;
        for (int64_t i = e0 + static_cast<int64_t>(threadIdx.x) * VEC; i < e1; i += 256 * VEC) {
            float u[VEC];
            load_u<G_BF16, HAS_H, VEC>(g, h, i, c.lam, u);
#pragma unroll
            for (int k = 0; k < VEC; ++k) acc = fmaf(u[k], u[k], acc);
        }
        acc = warp_sum_f(acc);
        if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = acc;
        __syncthreads();
        if (threadIdx.x == 0) {
            float tot = 0.0f;
#pragma unroll
            for (int w = 0; w < 8; ++w) tot += red[w];
            const float vv = fmaf(c.beta2, vb[b], c.one_m_beta2 * (tot / static_cast<float>(e1 - e0)));
            vb[b] = vv;
            s_den = sqrtf(vv * c.inv_bc2) + c.eps;
        }
        __syncthreads();
        const float den = s_den;
        for (int64_t i = e0 + static_cast<int64_t>(threadIdx.x) * VEC; i < e1; i += 256 * VEC) {
            float u[VEC];
            load_u<G_BF16, HAS_H, VEC>(g, h, i, c.lam, u);
            if constexpr (VEC == 4) {
                float4 th = __ldcs(reinterpret_cast<const float4*>(theta + i));
                th.x = apply_step(c.decay, th.x, c.lr, u[0] / den);
                th.y = apply_step(c.decay, th.y, c.lr, u[1] / den);
                th.z = apply_step(c.decay, th.z, c.lr, u[2] / den);
                th.w = apply_step(c.decay, th.w, c.lr, u[3] / den);
                __stcs(reinterpret_cast<float4*>(theta + i), th);
                if constexpr (SHADOW) {
                    uint2 sh;
                    sh.x = pack_bf16x2(th.x, th.y);
                    sh.y = pack_bf16x2(th.z, th.w);
                    __stcs(reinterpret_cast<uint2*>(shadow + i), sh);
                }
            } else {
#pragma unroll
                for (int k = 0; k < VEC; ++k) {
                    const float th = apply_step(c.decay, theta[i + k], c.lr, u[k] / den);
                    theta[i + k] = th;
                    if (SHADOW) reinterpret_cast<__nv_bfloat16*>(shadow)[i + k] = __float2bfloat16_rn(th);
                }
            }
        }
        __syncthreads();   // red and s_den are reused by the next block
    }
}

// Blocks of at most 8192 elements (d % 4 == 0): each of the CTA's NT threads
// keeps its WPT words of g (packed as loaded), h and theta in registers from
// one read, so a block costs one memory round trip before the reduction and
// none after it; v of the block is fetched with the data.  Blocks up to 4096
// elements use 256 threads and WPT 1, 2 or 4 (the smallest with
// 1024 WPT >= block, which keeps the registers, and so the resident CTAs
// whose loads hide the latency, matched to the block); larger ones use 512
// threads and WPT 4, so every block size keeps two register sets.
constexpr int kRegMaxBlock = 8192;
template <bool G_BF16>
struct GWord {
    using T = typename std::conditional<G_BF16, uint2, float4>::type;
};
template <bool G_BF16, bool HAS_H>
__device__ __forceinline__ void word_u(const typename GWord<G_BF16>::T& gw, const float4& hw, float lam,
                                       float (&u)[4]) {
    if constexpr (G_BF16) {
        u[0] = __uint_as_float(gw.x << 16);
        u[1] = __uint_as_float(gw.x & 0xFFFF0000u);
        u[2] = __uint_as_float(gw.y << 16);
        u[3] = __uint_as_float(gw.y & 0xFFFF0000u);
    } else {
        u[0] = gw.x; u[1] = gw.y; u[2] = gw.z; u[3] = gw.w;
    }
    if constexpr (HAS_H) {
        const float hv[4] = {hw.x, hw.y, hw.z, hw.w};
#pragma unroll
        for (int k = 0; k < 4; ++k) u[k] = (1.0f - lam) * u[k] + lam * hv[k];
    }
}

// One block's words of g, h and theta (and v_b in thread 0) in registers.
template <bool G_BF16, int WPT>
struct RowRegs {
    typename GWord<G_BF16>::T gw[WPT];
    float4 hw[WPT];
    float4 th[WPT];
    float vprev;
};

template <bool G_BF16, bool HAS_H, int WPT, int NT>
__device__ __forceinline__ void row_load(RowRegs<G_BF16, WPT>& r, const void* g, const float* h, const float* theta,
                                         const float* vb, int64_t b, int64_t block, int64_t n) {
    using GW = typename GWord<G_BF16>::T;
    const int64_t e0 = b * block;
    const int64_t e1 = e0 + block < n ? e0 + block : n;
    r.vprev = threadIdx.x == 0 ? vb[b] : 0.0f;
#pragma unroll
    for (int k = 0; k < WPT; ++k) {
        const int64_t i = e0 + 4 * (static_cast<int64_t>(threadIdx.x) + NT * k);
        if (i < e1) {
            r.gw[k] = *reinterpret_cast<const GW*>(static_cast<const char*>(g) + i * (G_BF16 ? 2 : 4));
            if constexpr (HAS_H) r.hw[k] = *reinterpret_cast<const float4*>(h + i);
            r.th[k] = __ldcs(reinterpret_cast<const float4*>(theta + i));
        }
    }
}

// Reduction, v_b and the update of block b from its registers.
template <bool G_BF16, bool HAS_H, bool SHADOW, int WPT, int NT>
__device__ __forceinline__ void row_update(const RowRegs<G_BF16, WPT>& r, float* theta, float* vb, uint16_t* shadow,
                                           int64_t b, int64_t block, int64_t n, const UpdCoef& c, float* red,
                                           float* s_den) {
    const int64_t e0 = b * block;
    const int64_t e1 = e0 + block < n ? e0 + block : n;
    float acc = 0.0f;
#pragma unroll
    for (int k = 0; k < WPT; ++k) {
        const int64_t i = e0 + 4 * (static_cast<int64_t>(threadIdx.x) + NT * k);
        if (i < e1) {
            float u[4];
            word_u<G_BF16, HAS_H>(r.gw[k], r.hw[k], c.lam, u);
#pragma unroll
            for (int q = 0; q < 4; ++q) acc = fmaf(u[q], u[q], acc);
        }
    }
    acc = warp_sum_f(acc);
    if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = acc;
    __syncthreads();
    if (threadIdx.x == 0) {
        float tot = 0.0f;
#pragma unroll
        for (int w = 0; w < NT / 32; ++w) tot += red[w];
        const float vv = fmaf(c.beta2, r.vprev, c.one_m_beta2 * (tot / static_cast<float>(e1 - e0)));
        vb[b] = vv;
        *s_den = sqrtf(vv * c.inv_bc2) + c.eps;
    }
    __syncthreads();
    const float den = *s_den;
#pragma unroll
    for (int k = 0; k < WPT; ++k) {
        const int64_t i = e0 + 4 * (static_cast<int64_t>(threadIdx.x) + NT * k);
        if (i < e1) {
            float u[4];
            word_u<G_BF16, HAS_H>(r.gw[k], r.hw[k], c.lam, u);
            float4 t = r.th[k];
            t.x = apply_step(c.decay, t.x, c.lr, u[0] / den);
            t.y = apply_step(c.decay, t.y, c.lr, u[1] / den);
            t.z = apply_step(c.decay, t.z, c.lr, u[2] / den);
            t.w = apply_step(c.decay, t.w, c.lr, u[3] / den);
            __stcs(reinterpret_cast<float4*>(theta + i), t);
            if constexpr (SHADOW) {
                uint2 sh;
                sh.x = pack_bf16x2(t.x, t.y);
                sh.y = pack_bf16x2(t.z, t.w);
                __stcs(reinterpret_cast<uint2*>(shadow + i), sh);
            }
        }
    }
    __syncthreads();   // red and s_den are reused by the next block
}

// The CTA walks its blocks b, b + grid, ... with two register sets: the
// loads of the next block are issued before the current one is reduced and
// written, so the CTA keeps a block's reads in flight through its barriers.
template <bool G_BF16, bool HAS_H, bool SHADOW, int WPT, int NT>
__global__ void __launch_bounds__(NT) update_blockshared_reg_kernel(float* __restrict__ theta,
                                                                    const void* __restrict__ g,
                                                                    const float* __restrict__ h,
                                                                    float* __restrict__ vb,
                                                                    uint16_t* __restrict__ shadow, int64_t n,
                                                                    int64_t block, UpdCoef c_in) {
    pdl_enter();
    __shared__ float red[NT / 32];
    __shared__ float s_den;
    const UpdCoef c = resolve_coef(c_in, nullptr);
    const int64_t nb = (n + block - 1) / block;
    const int64_t G = gridDim.x;
    int64_t b = blockIdx.x;
    if (b >= nb) return;
    RowRegs<G_BF16, WPT> ra, rb;
    row_load<G_BF16, HAS_H, WPT, NT>(ra, g, h, theta, vb, b, block, n);
    for (;;) {
        if (b + G < nb) row_load<G_BF16, HAS_H, WPT, NT>(rb, g, h, theta, vb, b + G, block, n);
        row_update<G_BF16, HAS_H, SHADOW, WPT, NT>(ra, theta, vb, shadow, b, block, n, c, red, &s_den);
        b += G;
        if (b >= nb) break;
        if (b + G < nb) row_load<G_BF16, HAS_H, WPT, NT>(ra, g, h, theta, vb, b + G, block, n);
        row_update<G_BF16, HAS_H, SHADOW, WPT, NT>(rb, theta, vb, shadow, b, block, n, c, red, &s_den);
        b += G;
        if (b >= nb) break;
    }
}

// Resident CTAs per SM times the SM count, at most the number of blocks.
template <typename K>
int resident_grid(K kernel, int64_t nb, int nt) {
    int per_sm = 0;
    if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kernel, nt, 0) != cudaSuccess || per_sm < 1)
        per_sm = 1;
    const int64_t grid = static_cast<int64_t>(device_sm_count()) * per_sm;
    return static_cast<int>(grid < nb ? grid : nb);
}

template <bool G_BF16, bool HAS_H, bool SHADOW, int WPT, int NT>
void launch_reg(float* theta, const void* g, const float* h, float* vb, uint16_t* shadow, int64_t n, int64_t block,
                const UpdCoef& c, cudaStream_t s) {
    auto k = update_blockshared_reg_kernel<G_BF16, HAS_H, SHADOW, WPT, NT>;
    launch_k(k, dim3(resident_grid(k, (n + block - 1) / block, NT)), dim3(NT), 0, s, theta, g, h, vb, shadow, n,
             block, c);
}

template <bool G_BF16, bool HAS_H, bool SHADOW>
void launch_reg_wpt(float* theta, const void* g, const float* h, float* vb, uint16_t* shadow, int64_t n,
                    int64_t block, const UpdCoef& c, cudaStream_t s) {
    if (block <= 1024) launch_reg<G_BF16, HAS_H, SHADOW, 1, 256>(theta, g, h, vb, shadow, n, block, c, s);
    else if (block <= 2048) launch_reg<G_BF16, HAS_H, SHADOW, 2, 256>(theta, g, h, vb, shadow, n, block, c, s);
    else if (block <= 4096) launch_reg<G_BF16, HAS_H, SHADOW, 4, 256>(theta, g, h, vb, shadow, n, block, c, s);
    else launch_reg<G_BF16, HAS_H, SHADOW, 4, 512>(theta, g, h, vb, shadow, n, block, c, s);
}

// Launch shape of the cluster kernel; at[] must hold two attributes.
template <bool G_BF16, bool HAS_H, bool SHADOW, int VEC>
cudaLaunchConfig_t cluster_cfg(cudaLaunchAttribute* at) {
    cudaLaunchConfig_t cfg = {};
    at[0].id = cudaLaunchAttributeClusterDimension;
    at[0].val.clusterDim.x = kBlockCluster;
    at[0].val.clusterDim.y = 1;
    at[0].val.clusterDim.z = 1;
    at[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    at[1].val.programmaticStreamSerializationAllowed = 1;
    cfg.blockDim = dim3(256);
    cfg.attrs = at;
    cfg.numAttrs = 2;
    return cfg;
}

// Clusters of the cluster kernel that run at once (cached per instantiation
// and device).
template <bool G_BF16, bool HAS_H, bool SHADOW, int VEC>
int cluster_slots() {
    constexpr int kMaxDev = 64;
    static std::atomic<int> slots_dev[kMaxDev];
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDev) {
        cudaGetLastError();
        dev = 0;
    }
    int slots = slots_dev[dev].load(std::memory_order_relaxed);
    if (slots == 0) {
        cudaLaunchAttribute at[2];
        cudaLaunchConfig_t cfg = cluster_cfg<G_BF16, HAS_H, SHADOW, VEC>(at);
        cfg.gridDim = dim3(static_cast<unsigned>(device_sm_count() / kBlockCluster * kBlockCluster));
        int m = 0;
        if (cudaOccupancyMaxActiveClusters(&m, update_blockshared_cluster_kernel<G_BF16, HAS_H, SHADOW, VEC>, &cfg) !=
                cudaSuccess ||
            m < 1) {
            cudaGetLastError();
            m = device_sm_count() / kBlockCluster;
        }
        slots = m > 0 ? m : 1;
        slots_dev[dev].store(slots, std::memory_order_relaxed);
    }
    return slots;
}

template <bool G_BF16, bool HAS_H, bool SHADOW, int VEC>
int launch_cluster(float* theta, const void* g, const float* h, float* vb, uint16_t* shadow, int64_t n,
                   int64_t block, const UpdCoef& c, int64_t nclusters, cudaStream_t s) {
    cudaLaunchAttribute at[2];
    cudaLaunchConfig_t cfg = cluster_cfg<G_BF16, HAS_H, SHADOW, VEC>(at);
    cfg.gridDim = dim3(static_cast<unsigned>(nclusters * kBlockCluster));
    cfg.stream = s;
    cudaLaunchKernelEx(&cfg, update_blockshared_cluster_kernel<G_BF16, HAS_H, SHADOW, VEC>, theta, g, h, vb, shadow,
                       n, block, c);
    count_launch();
    return BOM_OK;
}

// A stream-ordered memory pool of the library's own on the current device,
// kept reserved between calls (release threshold at its maximum), so the few
// KB of scratch below cost no mapping after the first call and calls on
// different streams never share a buffer.
cudaMemPool_t scratch_pool() {
    static std::mutex mu;
    static cudaMemPool_t pools[64] = {};
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return nullptr;
    std::lock_guard<std::mutex> lock(mu);
    if (pools[dev] == nullptr) {
        cudaMemPoolProps props = {};
        props.allocType = cudaMemAllocationTypePinned;
        props.handleTypes = cudaMemHandleTypeNone;
        props.location.type = cudaMemLocationTypeDevice;
        props.location.id = dev;
        cudaMemPool_t pool = nullptr;
        if (cudaMemPoolCreate(&pool, &props) != cudaSuccess) {
            cudaGetLastError();
            return nullptr;
        }
        uint64_t keep = ~uint64_t(0);
        cudaMemPoolSetAttribute(pool, cudaMemPoolAttrReleaseThreshold, &keep);
        pools[dev] = pool;
    }
    return pools[dev];
}

// The grid-wide path; its partials and denominators live in a stream-ordered
// scratch of (chunks + blocks) floats from scratch_pool, freed on the same
// stream.
template <bool G_BF16, bool HAS_H, bool SHADOW, int VEC>
int launch_grid_blocks(float* theta, const void* g, const float* h, float* vb, uint16_t* shadow, int64_t n,
                       int64_t block, const UpdCoef& c, cudaStream_t s) {
    const int64_t nb = (n + block - 1) / block;
    const int64_t G = 4 * static_cast<int64_t>(device_sm_count());
    int64_t S = (4 * G + nb - 1) / nb;                 // chunks per block: about four per CTA in all
    int64_t ch = (block + S - 1) / S;
    ch = (ch + 1023) / 1024 * 1024;                    // whole passes of 256 threads x 4 elements
    S = (block + ch - 1) / ch;
    const int64_t nchunks = nb * S;
    float* scr = nullptr;
    cudaMemPool_t pool = scratch_pool();
    if (pool == nullptr || cudaMallocFromPoolAsync(reinterpret_cast<void**>(&scr),
                                                   static_cast<size_t>(nchunks + nb) * sizeof(float), pool, s) !=
                               cudaSuccess) {
        cudaGetLastError();
        return BOM_ENOMEM;
    }
    float* part = scr;
    float* den = scr + nchunks;
    const int64_t g1 = nchunks < G ? nchunks : G;
    launch_k(bs_chunk_sq_kernel<G_BF16, HAS_H, VEC>, dim3(static_cast<unsigned>(g1)), dim3(256), 0, s, g, h, c.lam, n, block, ch, S,
                                                                                    nchunks, part);
    count_launch();
    launch_k(bs_finish_kernel, dim3(static_cast<unsigned>((nb + 7) / 8)), dim3(256), 0, s, part, S, nb, n, block, vb, den, c);
    count_launch();
    const int64_t need = (n / VEC + 255) / 256;
    int64_t g3 = 8 * static_cast<int64_t>(device_sm_count());
    if (g3 > need) g3 = need;
    if (g3 < 1) g3 = 1;
    launch_k(bs_apply_kernel<G_BF16, HAS_H, SHADOW, VEC>, dim3(static_cast<unsigned>(g3)), dim3(256), 0, s, theta, g, h, shadow, n,
                                                                                          block, den, c);
    count_launch();
    cudaFreeAsync(scr, s);
    return BOM_OK;
}

// Blocks above the register-resident size: the cluster kernel when there are
// enough blocks to occupy every cluster slot, else the grid-wide path.
template <bool G_BF16, bool HAS_H, bool SHADOW, int VEC>
int launch_large_blocks(float* theta, const void* g, const float* h, float* vb, uint16_t* shadow, int64_t n,
                        int64_t block, const UpdCoef& c, cudaStream_t s) {
    const int64_t nb = (n + block - 1) / block;
    const int64_t slots = cluster_slots<G_BF16, HAS_H, SHADOW, VEC>();
    if (nb >= slots) return launch_cluster<G_BF16, HAS_H, SHADOW, VEC>(theta, g, h, vb, shadow, n, block, c, slots, s);
    return launch_grid_blocks<G_BF16, HAS_H, SHADOW, VEC>(theta, g, h, vb, shadow, n, block, c, s);
}

template <bool G_BF16, bool HAS_H, int VEC>
int dispatch_blockshared(float* theta, const void* g, const float* h, float* vb, uint16_t* shadow, int64_t n,
                         int64_t block, const UpdCoef& c, int grid, cudaStream_t s) {
    if (block > kRegMaxBlock) {
        if (shadow) return launch_large_blocks<G_BF16, HAS_H, true, VEC>(theta, g, h, vb, shadow, n, block, c, s);
        return launch_large_blocks<G_BF16, HAS_H, false, VEC>(theta, g, h, vb, shadow, n, block, c, s);
    }
    if (VEC == 4) {
        if (shadow) launch_reg_wpt<G_BF16, HAS_H, true>(theta, g, h, vb, shadow, n, block, c, s);
        else launch_reg_wpt<G_BF16, HAS_H, false>(theta, g, h, vb, shadow, n, block, c, s);
    } else if (shadow) {
        launch_k(update_blockshared_kernel<G_BF16, HAS_H, true, VEC>, dim3(grid), dim3(256), 0, s, theta, g, h, vb, shadow, n, block, c);
    } else {
        launch_k(update_blockshared_kernel<G_BF16, HAS_H, false, VEC>, dim3(grid), dim3(256), 0, s, theta, g, h, vb, shadow, n, block,
                                                                                  c);
    }
    count_launch();
    return BOM_OK;
}

template <bool G_BF16, bool HAS_H>
void dispatch_shadow(float* theta, const void* g, const float* h, float* v, uint16_t* shadow, int64_t n,
                     const UpdCoef& c, int grid, const double* clip_sq, float max_norm, const DevScalars* sc,
                     cudaStream_t s) {
    if (clip_sq) {
        if (shadow)
            launch_k(update_kernel<G_BF16, HAS_H, true, true>, dim3(grid), dim3(256), 0, s, theta, g, h, v, shadow, n, c, clip_sq,
                                                                          max_norm, sc);
        else
            launch_k(update_kernel<G_BF16, HAS_H, false, true>, dim3(grid), dim3(256), 0, s, theta, g, h, v, shadow, n, c, clip_sq,
                                                                           max_norm, sc);
    } else {
        if (shadow)
            launch_k(update_kernel<G_BF16, HAS_H, true, false>, dim3(grid), dim3(256), 0, s, theta, g, h, v, shadow, n, c, nullptr,
                                                                           0.0f, sc);
        else
            launch_k(update_kernel<G_BF16, HAS_H, false, false>, dim3(grid), dim3(256), 0, s, theta, g, h, v, shadow, n, c, nullptr,
                                                                            0.0f, sc);
    }
    count_launch();
}

// sum u^2 over a flat range: per-thread fp32 sums, per-block fp64 partials in
// fixed slots, then one block adds them in order to *sq.
template <bool G_BF16, bool HAS_H>
__global__ void __launch_bounds__(256) sqnorm_part_kernel(const void* __restrict__ g, const float* __restrict__ h,
                                                          float lam, int64_t n, double* __restrict__ part) {
    pdl_enter();
    float acc = 0.0f;
    const int64_t n4 = n >> 2;
    const int64_t stride = static_cast<int64_t>(gridDim.x) * blockDim.x;
    for (int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; i < n4; i += stride) {
        float u[4];
        load_u<G_BF16, HAS_H, 4>(g, h, 4 * i, lam, u);
#pragma unroll
        for (int k = 0; k < 4; ++k) acc = fmaf(u[k], u[k], acc);
    }
    if (blockIdx.x == 0 && threadIdx.x < (n & 3)) {
        float u[1];
        load_u<G_BF16, HAS_H, 1>(g, h, (n4 << 2) + threadIdx.x, lam, u);
        acc = fmaf(u[0], u[0], acc);
    }
    __shared__ float red[8];
    acc = warp_sum_f(acc);
    if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = acc;
    __syncthreads();
    if (threadIdx.x == 0) {
        double t = 0.0;
        for (int w = 0; w < 8; ++w) t += static_cast<double>(red[w]);
        part[blockIdx.x] = t;
    }
}

// *sq += sum_b part[b]: lane l adds blocks l, l + 32, ... in order, then a
// fixed shuffle tree (the order depends only on nblocks: deterministic).
__global__ void sqnorm_finish_kernel(const double* __restrict__ part, int nblocks, double* __restrict__ sq) {
    pdl_enter();
    const int l = threadIdx.x & 31;
    double t = 0.0;
    for (int b = l; b < nblocks; b += 32) t += part[b];
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) t += __shfl_xor_sync(0xffffffffu, t, o);
    if (threadIdx.x == 0) *sq += t;
}

}  // namespace

int launch_update(float* theta, const void* g, int g_bf16, const float* h, float* v, uint16_t* shadow, int64_t n,
                  float lr, float wd, float lambda, float beta2, float eps, float inv_bc2, const double* clip_sq,
                  float max_norm, const DevScalars* sc, cudaStream_t s, bool step_scalars) {
    if (n <= 0) return BOM_OK;
    UpdCoef c;
    c.lr = lr;
    c.wd = wd;
    c.decay = 0.0f;
    c.from_step = step_scalars ? 1 : 0;
    c.lam = lambda;
    c.beta2 = beta2;
    c.one_m_beta2 = 1.0f - beta2;
    c.eps = eps;
    c.inv_bc2 = inv_bc2;
    const int64_t n4 = (n >> 2) > 0 ? (n >> 2) : 1;
    int64_t grid = static_cast<int64_t>(device_sm_count()) * 8;
    const int64_t need = (n4 + 255) / 256;
    if (grid > need) grid = need;
    if (grid < 1) grid = 1;
    if (g_bf16) {
        if (h) dispatch_shadow<true, true>(theta, g, h, v, shadow, n, c, (int)grid, clip_sq, max_norm, sc, s);
        else dispatch_shadow<true, false>(theta, g, h, v, shadow, n, c, (int)grid, clip_sq, max_norm, sc, s);
    } else {
        if (h) dispatch_shadow<false, true>(theta, g, h, v, shadow, n, c, (int)grid, clip_sq, max_norm, sc, s);
        else dispatch_shadow<false, false>(theta, g, h, v, shadow, n, c, (int)grid, clip_sq, max_norm, sc, s);
    }
    return cudaPeekAtLastError() == cudaSuccess ? BOM_OK : BOM_ECUDA;
}

namespace {

// BOM-AdamW update of several tensors in one launch (the update after a small
// step's weight gradients; see launch_update_multi).  Each tensor's elements
// are walked as 16-byte words (fp32 theta, v and u; bf16 compute copy), the
// tensors one after another in a single grid-stride range.
struct MultiUpdTable {
    int ntensor;
    int copy_f32;                      // compute copies in fp32 (else bf16)
    int64_t word0[kMultiUpdMax + 1];   // first word of each tensor in the joint range
    float* theta[kMultiUpdMax];
    float* v[kMultiUpdMax];
    const float* u[kMultiUpdMax];
    void* copy[kMultiUpdMax];
    int64_t n[kMultiUpdMax];
    float wd[kMultiUpdMax];
    // a bias whose u is the column sum of a cotangent: u_j = sum_i src[i, j]
    // over `rows` rows in order (src [rows, n]: the cotangent in the compute
    // dtype, or fp32 column sums of its 32-row blocks), else null
    const void* src[kMultiUpdMax];
    int64_t rows[kMultiUpdMax];
    int src_f32[kMultiUpdMax];
};

__global__ void __launch_bounds__(256) update_multi_kernel(const __grid_constant__ MultiUpdTable tb, UpdCoef c_in,
                                                           const DevScalars* sc, int64_t* t_adv) {
    pdl_enter();
    if (sc != nullptr && sc->status != 0) return;
    // the step succeeded: advance the device step counter (nothing in this
    // launch reads it; the next step's kernels start after this one ends)
    if (t_adv != nullptr && blockIdx.x == 0 && threadIdx.x == 0) *t_adv += 1;
    const int64_t words = tb.word0[tb.ntensor];
    const int64_t stride = static_cast<int64_t>(gridDim.x) * blockDim.x;
    int k = 0;
    for (int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; i < words; i += stride) {
        while (i >= tb.word0[k + 1]) ++k;   // words only increase along a thread's walk
        UpdCoef c = c_in;
        c.wd = tb.wd[k];
        c = resolve_coef(c, sc);
        const int64_t w = i - tb.word0[k];
        const int64_t e0 = 4 * w;
        const int64_t len = tb.n[k];
        if (tb.src[k] != nullptr && tb.src_f32[k] && e0 + 4 <= len && (len & 3) == 0 &&
            (reinterpret_cast<uintptr_t>(tb.src[k]) & 15u) == 0) {
            // a bias whose u sums fp32 rows (16-byte aligned rows): the word's four
            // columns at once, every row load and theta, v in flight together;
            // per column the same order of additions as the loop below
            const float4* sp = static_cast<const float4*>(tb.src[k]) + w;
            const int64_t rstride = len / 4;
            float4 th = __ldcs(reinterpret_cast<const float4*>(tb.theta[k]) + w);
            float4 vv = __ldcs(reinterpret_cast<const float4*>(tb.v[k]) + w);
            float4 a8[8];
#pragma unroll
            for (int q = 0; q < 8; ++q) a8[q] = make_float4(0.0f, 0.0f, 0.0f, 0.0f);
            const int64_t rows = tb.rows[k];
            int64_t r = 0;
            for (; r + 8 <= rows; r += 8) {
                float4 x[8];
#pragma unroll
                for (int q = 0; q < 8; ++q) x[q] = sp[(r + q) * rstride];
#pragma unroll
                for (int q = 0; q < 8; ++q) {
                    a8[q].x += x[q].x;
                    a8[q].y += x[q].y;
                    a8[q].z += x[q].z;
                    a8[q].w += x[q].w;
                }
            }
#pragma unroll
            for (int q = 0; q < 8; ++q)
                if (r + q < rows) {
                    const float4 x = sp[(r + q) * rstride];
                    a8[q].x += x.x;
                    a8[q].y += x.y;
                    a8[q].z += x.z;
                    a8[q].w += x.w;
                }
            float4 u = make_float4(0.0f, 0.0f, 0.0f, 0.0f);
#pragma unroll
            for (int q = 0; q < 8; ++q) {
                u.x += a8[q].x;
                u.y += a8[q].y;
                u.z += a8[q].z;
                u.w += a8[q].w;
            }
            upd1(th.x, vv.x, u.x, c);
            upd1(th.y, vv.y, u.y, c);
            upd1(th.z, vv.z, u.z, c);
            upd1(th.w, vv.w, u.w, c);
            reinterpret_cast<float4*>(tb.theta[k])[w] = th;
            reinterpret_cast<float4*>(tb.v[k])[w] = vv;
            for (int j = 0; j < 4; ++j) st_elem(tb.copy[k], e0 + j, tb.copy_f32, j == 0 ? th.x : j == 1 ? th.y : j == 2 ? th.z : th.w);
        } else if (tb.src[k] != nullptr) {   // a bias: u from the column sums of its cotangent
            const int f32 = tb.src_f32[k];
            for (int64_t e = e0; e < e0 + 4 && e < len; ++e) {
                // rows r = 8q + w in eight interleaved sums, then w = 0..7 in
                // order: the order of the step's column reduction over one
                // range of at most 128 rows, so both give the same bits there
                float a8[8];
#pragma unroll
                for (int q = 0; q < 8; ++q) a8[q] = 0.0f;
                const int64_t rows = tb.rows[k];
                int64_t r = 0;
                for (; r + 8 <= rows; r += 8) {
                    float x[8];
#pragma unroll
                    for (int q = 0; q < 8; ++q) x[q] = ld_elem(tb.src[k], (r + q) * len + e, f32);
#pragma unroll
                    for (int q = 0; q < 8; ++q) a8[q] += x[q];
                }
#pragma unroll
                for (int q = 0; q < 8; ++q)
                    if (r + q < rows) a8[q] += ld_elem(tb.src[k], (r + q) * len + e, f32);
                float u = 0.0f;
#pragma unroll
                for (int q = 0; q < 8; ++q) u += a8[q];
                float th = tb.theta[k][e], vv = tb.v[k][e];
                upd1(th, vv, u, c);
                tb.theta[k][e] = th;
                tb.v[k][e] = vv;
                st_elem(tb.copy[k], e, tb.copy_f32, th);
            }
        } else if (e0 + 4 <= len) {
            float4 th = __ldcs(reinterpret_cast<const float4*>(tb.theta[k]) + w);
            float4 vv = __ldcs(reinterpret_cast<const float4*>(tb.v[k]) + w);
            const float4 u = __ldcs(reinterpret_cast<const float4*>(tb.u[k]) + w);
            upd1(th.x, vv.x, u.x, c);
            upd1(th.y, vv.y, u.y, c);
            upd1(th.z, vv.z, u.z, c);
            upd1(th.w, vv.w, u.w, c);
            __stcs(reinterpret_cast<float4*>(tb.theta[k]) + w, th);
            __stcs(reinterpret_cast<float4*>(tb.v[k]) + w, vv);
            if (tb.copy_f32) {
                __stcs(reinterpret_cast<float4*>(tb.copy[k]) + w, th);
            } else {
                uint2 sh;
                sh.x = pack_bf16x2(th.x, th.y);
                sh.y = pack_bf16x2(th.z, th.w);
                __stcs(reinterpret_cast<uint2*>(tb.copy[k]) + w, sh);
            }
        } else {
            for (int64_t e = e0; e < len; ++e) {
                float th = tb.theta[k][e], vv = tb.v[k][e];
                upd1(th, vv, tb.u[k][e], c);
                tb.theta[k][e] = th;
                tb.v[k][e] = vv;
                st_elem(tb.copy[k], e, tb.copy_f32, th);
            }
        }
    }
}

}  // namespace

int launch_update_multi(int ntensor, float* const* theta, float* const* v, const float* const* u, void* const* copy,
                        int copy_f32, const int64_t* n, const float* wd, const void* const* src, const int64_t* rows,
                        const int* src_f32, float beta2, float eps, const DevScalars* sc, int64_t* t_adv,
                        cudaStream_t s) {
    if (ntensor < 1 || ntensor > kMultiUpdMax) return BOM_EINVAL;
    MultiUpdTable tb = {};
    tb.ntensor = ntensor;
    tb.copy_f32 = copy_f32;
    int64_t words = 0;
    for (int k = 0; k < ntensor; ++k) {
        tb.word0[k] = words;
        tb.theta[k] = theta[k];
        tb.v[k] = v[k];
        tb.u[k] = u[k];
        tb.copy[k] = copy[k];
        tb.n[k] = n[k];
        tb.wd[k] = wd[k];
        tb.src[k] = src ? src[k] : nullptr;
        tb.rows[k] = rows ? rows[k] : 0;
        tb.src_f32[k] = src_f32 ? src_f32[k] : copy_f32;
        words += (n[k] + 3) / 4;
    }
    tb.word0[ntensor] = words;
    UpdCoef c = {};
    c.from_step = 1;   // lr and 1/(1 - beta2^t) from the step scalars
    c.beta2 = beta2;
    c.one_m_beta2 = 1.0f - beta2;
    c.eps = eps;
    int64_t grid = static_cast<int64_t>(device_sm_count()) * 8;
    const int64_t need = (words + 255) / 256;
    if (grid > need) grid = need;
    if (grid < 1) grid = 1;
    launch_k(update_multi_kernel, dim3(static_cast<unsigned>(grid)), dim3(256), 0, s, tb, c, sc, t_adv);
    count_launch();
    return cudaPeekAtLastError() == cudaSuccess ? BOM_OK : BOM_ECUDA;
}

int sqnorm_blocks(int64_t n) {
    int64_t b = static_cast<int64_t>(device_sm_count()) * 4;
    const int64_t need = ((n >> 2) + 255) / 256;
    if (b > need) b = need;
    if (b > kOwnStepMaxBlocks) b = kOwnStepMaxBlocks;
    return static_cast<int>(b < 1 ? 1 : b);
}

int launch_sqnorm(const void* g, int g_bf16, const float* h, float lambda, int64_t n, double* part, double* sq,
                  cudaStream_t s) {
    if (n <= 0) return BOM_OK;
    const int nb = sqnorm_blocks(n);
    if (g_bf16) {
        if (h) launch_k(sqnorm_part_kernel<true, true>, dim3(nb), dim3(256), 0, s, g, h, lambda, n, part);
        else launch_k(sqnorm_part_kernel<true, false>, dim3(nb), dim3(256), 0, s, g, h, lambda, n, part);
    } else {
        if (h) launch_k(sqnorm_part_kernel<false, true>, dim3(nb), dim3(256), 0, s, g, h, lambda, n, part);
        else launch_k(sqnorm_part_kernel<false, false>, dim3(nb), dim3(256), 0, s, g, h, lambda, n, part);
    }
    count_launch();
    launch_k(sqnorm_finish_kernel, dim3(1), dim3(32), 0, s, part, nb, sq);
    count_launch();
    return cudaPeekAtLastError() == cudaSuccess ? BOM_OK : BOM_ECUDA;
}

int launch_update_blockshared(float* theta, const void* g, int g_bf16, const float* h, float* vb, uint16_t* shadow,
                              int64_t n, int64_t block, float lr, float wd, float lambda, float beta2, float eps,
                              float inv_bc2, cudaStream_t s) {
    if (n <= 0) return BOM_OK;
    UpdCoef c;
    c.lr = lr;
    c.wd = wd;
    c.decay = 0.0f;
    c.from_step = 0;
    c.lam = lambda;
    c.beta2 = beta2;
    c.one_m_beta2 = 1.0f - beta2;
    c.eps = eps;
    c.inv_bc2 = inv_bc2;
    const int64_t nb = (n + block - 1) / block;
    int64_t grid = static_cast<int64_t>(device_sm_count()) * 8;
    if (grid > nb) grid = nb;
    const bool vec = (block % 4 == 0) && (n % 4 == 0);
    const int gi = static_cast<int>(grid);
    int rc = BOM_OK;
    if (vec) {
        if (g_bf16) {
            if (h) rc = dispatch_blockshared<true, true, 4>(theta, g, h, vb, shadow, n, block, c, gi, s);
            else rc = dispatch_blockshared<true, false, 4>(theta, g, h, vb, shadow, n, block, c, gi, s);
        } else {
            if (h) rc = dispatch_blockshared<false, true, 4>(theta, g, h, vb, shadow, n, block, c, gi, s);
            else rc = dispatch_blockshared<false, false, 4>(theta, g, h, vb, shadow, n, block, c, gi, s);
        }
    } else {
        if (g_bf16) {
            if (h) rc = dispatch_blockshared<true, true, 1>(theta, g, h, vb, shadow, n, block, c, gi, s);
            else rc = dispatch_blockshared<true, false, 1>(theta, g, h, vb, shadow, n, block, c, gi, s);
        } else {
            if (h) rc = dispatch_blockshared<false, true, 1>(theta, g, h, vb, shadow, n, block, c, gi, s);
            else rc = dispatch_blockshared<false, false, 1>(theta, g, h, vb, shadow, n, block, c, gi, s);
        }
    }
    if (rc != BOM_OK) return rc;
    return cudaPeekAtLastError() == cudaSuccess ? BOM_OK : BOM_ECUDA;
}

}  // namespace bom
