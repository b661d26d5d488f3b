// tcgen05 GEMM engine for sm_103a: bf16 operands, fp32 accumulation in TMEM.
//
// One persistent CTA per SM walks the output tiles (128 x 256, or 128 x 128
// output columns when the B tile is split between gate and up weights).
// Warp roles:
//   warp 0     one thread issues TMA tile loads (128-byte swizzle) into a
//              4-stage shared-memory ring guarded by mbarriers;
//   warp 1     allocates 512 TMEM columns (two 128 x 256 fp32 accumulators)
//              and one thread issues the UMMAs (M = 128, N = 256, K = 16),
//              releasing each smem stage with tcgen05.commit;
//   warps 2-9  epilogue: tcgen05.ld of the accumulator (one TMEM lane = one
//              output row per thread; two warps per lane quarter, one per
//              column half), the fused epilogue of the step, and global
//              stores.  With two accumulators the epilogue of tile i overlaps
//              the mainloop of tile i+1.
// Every mbarrier wait is bounded; a wait that runs out latches BOM_ETIMEOUT,
// all roles unwind, in-flight TMA loads and UMMAs are drained, TMEM is freed.
#include <cstdio>
#include <mutex>

#include <cuda.h>
#include <cudaTypedefs.h>

#include "gemm.h"
#include "tc_ptx.cuh"

namespace bom {
namespace tc {

constexpr int BM = 128;
constexpr int BN = 256;
constexpr int BK = 64;  // one 128-byte swizzle atom of bf16 along K
constexpr int STAGES = 4;
constexpr int A_STAGE_BYTES = BM * BK * 2;  // 16 KB
constexpr int B_STAGE_BYTES = BN * BK * 2;  // 32 KB
constexpr int NUM_THREADS = 320;  // producer warp, UMMA warp, 8 epilogue warps
constexpr int TMEM_COLS = 512;
constexpr int SMEM_BYTES = STAGES * (A_STAGE_BYTES + B_STAGE_BYTES) + 1024 + 256;
constexpr int GROUP_M = 8;

struct Params {
    CUtensorMap mapA[2];
    CUtensorMap mapB[2];
    int M, N;
    int kb[2];
    int nseg;
    int tiles_m, tiles_n;
    int dual_b;
    int bn_out;
    EpiParams epi;
};

__device__ __forceinline__ void tile_coords(int tile, int tiles_m, int tiles_n, int& mt, int& nt) {
    const int per_group = GROUP_M * tiles_n;
    const int g = tile / per_group;
    const int first_m = g * GROUP_M;
    const int gsz = min(tiles_m - first_m, GROUP_M);
    const int r = tile - g * per_group;
    mt = first_m + r % gsz;
    nt = r / gsz;
}

// One 32-column chunk of a bf16 epilogue operand row (zeros past N) into
// words pk[4*slot .. 4*slot+3].
template <int NW>
__device__ __forceinline__ void load_chunk_bf16(const void* base, int64_t row_off, int n, int N, uint4 (&pk)[NW],
                                                int slot) {
    const uint16_t* p = static_cast<const uint16_t*>(base) + row_off + n;
    if (n + 32 <= N) {
#pragma unroll
        for (int i = 0; i < 4; ++i) pk[4 * slot + i] = __ldg(reinterpret_cast<const uint4*>(p) + i);
    } else {
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            uint32_t w[4];
#pragma unroll
            for (int j = 0; j < 4; ++j) {
                const int c = 8 * i + 2 * j;
                const uint32_t lo = (n + c < N) ? p[c] : 0u;
                const uint32_t hi = (n + c + 1 < N) ? p[c + 1] : 0u;
                w[j] = lo | (hi << 16);
            }
            pk[4 * slot + i] = make_uint4(w[0], w[1], w[2], w[3]);
        }
    }
}

// The 32 values held in words pk[4*slot .. 4*slot+3].
template <int NW>
__device__ __forceinline__ void unpack32_dyn(const uint4 (&pk)[NW], int slot, float (&v)[32]) {
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        const uint4 w = pk[4 * slot + i];
        const uint32_t ws[4] = {w.x, w.y, w.z, w.w};
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            v[8 * i + 2 * j] = __uint_as_float(ws[j] << 16);
            v[8 * i + 2 * j + 1] = __uint_as_float(ws[j] & 0xFFFF0000u);
        }
    }
}

__device__ __forceinline__ float fast_exp(float x) { return exp2f(x * 1.4426950408889634f); }
__device__ __forceinline__ float fast_sigmoid(float x) { return __frcp_rn(1.0f + fast_exp(-x)); }

__device__ __forceinline__ void tmem_load32(uint32_t taddr, float (&v)[32]) {
    uint32_t r[32];
    __syncwarp();
    tmem_ld_32x32b_x32(taddr, r);
    tmem_ld_wait();
#pragma unroll
    for (int i = 0; i < 32; ++i) v[i] = __uint_as_float(r[i]);
}

template <bool A_MN, bool B_MN, int EPI>
__global__ void __launch_bounds__(NUM_THREADS, 1) gemm_kernel(const __grid_constant__ Params p) {
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    uint8_t* sA = smem;
    uint8_t* sB = smem + STAGES * A_STAGE_BYTES;
    uint64_t* bars = reinterpret_cast<uint64_t*>(sB + STAGES * B_STAGE_BYTES);
    uint64_t* full = bars;
    uint64_t* empty = bars + STAGES;
    uint64_t* tfull = bars + 2 * STAGES;
    uint64_t* tempty = tfull + 2;
    uint64_t* drain = tempty + 2;
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(drain + 1);
    volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);
    int* skip_flag = reinterpret_cast<int*>(tmem_slot + 2);

    const int warp = threadIdx.x >> 5;
    const int lane = threadIdx.x & 31;

    if (threadIdx.x == 0) {
        for (int s = 0; s < STAGES; ++s) {
            mbar_init(&full[s], 1);
            mbar_init(&empty[s], 1);
        }
        for (int a = 0; a < 2; ++a) {
            mbar_init(&tfull[a], 1);
            mbar_init(&tempty[a], 256);
        }
        mbar_init(drain, 1);
        *abort_flag = 0;
        *skip_flag = (p.epi.sc != nullptr && p.epi.sc->status != 0) ? 1 : 0;
        fence_barrier_init();
    }
    if (warp == 0 && lane == 0) {
        prefetch_tensormap(&p.mapA[0]);
        prefetch_tensormap(&p.mapB[0]);
    }
    if (warp == 1) {
        tmem_alloc(tmem_slot, TMEM_COLS);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem_base = *tmem_slot;
    const bool skip = *skip_flag != 0;

    const int num_tiles = p.tiles_m * p.tiles_n;
    const int kb_total = p.kb[0] + (p.nseg > 1 ? p.kb[1] : 0);

    if (!skip && warp == 0) {
        // ------------------------------------------------------------ TMA producer
        if (lane == 0 && kb_total > 0) {
            int stage = 0;
            uint32_t phase = 0;
            uint32_t issued_mask = 0, issued_phase = 0;
            bool ok = true;
            for (int tile = blockIdx.x; ok && tile < num_tiles; tile += gridDim.x) {
                int mt, nt;
                tile_coords(tile, p.tiles_m, p.tiles_n, mt, nt);
                const int m0 = mt * BM;
                const int n0 = nt * p.bn_out;
                for (int seg = 0; ok && seg < p.nseg; ++seg) {
                    for (int kb = 0; kb < p.kb[seg]; ++kb) {
                        if (!mbar_wait_bounded(&empty[stage], phase ^ 1u, abort_flag)) {
                            ok = false;
                            break;
                        }
                        mbar_arrive_expect_tx(&full[stage], A_STAGE_BYTES + B_STAGE_BYTES);
                        const int k0 = kb * BK;
                        uint8_t* a = sA + stage * A_STAGE_BYTES;
                        uint8_t* b = sB + stage * B_STAGE_BYTES;
                        if (!A_MN) {
                            tma_load_2d(a, &p.mapA[seg], &full[stage], k0, m0);
                        } else {
                            tma_load_2d(a, &p.mapA[seg], &full[stage], m0, k0);
                            tma_load_2d(a + 8192, &p.mapA[seg], &full[stage], m0 + 64, k0);
                        }
                        if (p.dual_b) {
                            tma_load_2d(b, &p.mapB[0], &full[stage], k0, n0);
                            tma_load_2d(b + 16384, &p.mapB[1], &full[stage], k0, n0);
                        } else if (!B_MN) {
                            tma_load_2d(b, &p.mapB[seg], &full[stage], k0, n0);
                        } else {
#pragma unroll
                            for (int j = 0; j < 4; ++j)
                                tma_load_2d(b + j * 8192, &p.mapB[seg], &full[stage], n0 + 64 * j, k0);
                        }
                        issued_mask |= 1u << stage;
                        issued_phase = (issued_phase & ~(1u << stage)) | (phase << stage);
                        if (++stage == STAGES) {
                            stage = 0;
                            phase ^= 1u;
                        }
                    }
                }
            }
            // Every issued load must land before the CTA may exit.
            for (int s = 0; s < STAGES; ++s)
                if (issued_mask & (1u << s)) mbar_wait_bounded(&full[s], (issued_phase >> s) & 1u, nullptr);
        }
    } else if (!skip && warp == 1) {
        // ------------------------------------------------------------ UMMA issuer
        if (lane == 0 && kb_total > 0) {
            constexpr uint32_t idesc = idesc_bf16_f32(BM, BN, A_MN, B_MN);
            int stage = 0;
            uint32_t phase = 0;
            bool ok = true;
            int it = 0;
            for (int tile = blockIdx.x; ok && tile < num_tiles; tile += gridDim.x, ++it) {
                const int acc = it & 1;
                const uint32_t aph = (it >> 1) & 1;
                if (!mbar_wait_bounded(&tempty[acc], aph ^ 1u, abort_flag)) break;
                tc_fence_after();
                const uint32_t d_tmem = tmem_base + static_cast<uint32_t>(acc * BN);
                for (int kb = 0; kb < kb_total; ++kb) {
                    if (!mbar_wait_bounded(&full[stage], phase, abort_flag)) {
                        ok = false;
                        break;
                    }
                    tc_fence_after();
                    const uint32_t a0 = smem_u32(sA + stage * A_STAGE_BYTES);
                    const uint32_t b0 = smem_u32(sB + stage * B_STAGE_BYTES);
#pragma unroll
                    for (int kk = 0; kk < BK / 16; ++kk) {
                        const uint64_t ad = A_MN ? smem_desc_sw128(a0 + kk * 2048, 8192, 1024)
                                                 : smem_desc_sw128(a0 + kk * 32, 16, 1024);
                        const uint64_t bd = B_MN ? smem_desc_sw128(b0 + kk * 2048, 8192, 1024)
                                                 : smem_desc_sw128(b0 + kk * 32, 16, 1024);
                        umma_bf16(d_tmem, ad, bd, idesc, (kb | kk) != 0 ? 1u : 0u);
                    }
                    umma_commit(&empty[stage]);
                    if (++stage == STAGES) {
                        stage = 0;
                        phase ^= 1u;
                    }
                }
                if (ok) umma_commit(&tfull[acc]);
            }
            // All issued UMMAs must finish before TMEM is released.
            umma_commit(drain);
            mbar_wait_bounded(drain, 0, nullptr);
        }
    } else if (!skip && warp >= 2) {
        // ------------------------------------------------------------ epilogue
        // Eight warps: warp w reads TMEM lane quarter (w & 3) (its 32 output
        // rows) and column half h of the tile, so every TMEM quarter has two
        // warps and the epilogue's global-memory latency is overlapped twice.
        const int q = warp & 3;
        const int h = (warp - 2) >> 2;
        const int row = q * 32 + lane;
        const EpiParams& e = p.epi;
        constexpr int CPW = BN / 64;  // 32-column chunks per warp
        int it = 0;
        for (int tile = blockIdx.x; tile < num_tiles; tile += gridDim.x, ++it) {
            int mt, nt;
            tile_coords(tile, p.tiles_m, p.tiles_n, mt, nt);
            const int m0 = mt * BM;
            const int n0 = nt * p.bn_out;
            const int acc = it & 1;
            const int m = m0 + row;
            const bool valid = m < p.M;
            const int c0 = h * CPW;
            // Per-row epilogue operands do not depend on the accumulator: the
            // warp's first chunk is loaded before the mainloop wait, and each
            // later chunk while the previous one is being processed.
            uint4 xa[4], xb[4];
            const bool has_a = valid && ((EPI == EPI_SWIGLU_BWD) || (EPI == EPI_LINEAR && e.resid != nullptr));
            const bool has_b = valid && ((EPI == EPI_SWIGLU_BWD) || (EPI == EPI_LINEAR && e.act == ACT_DGELU));
            const void* pa = EPI == EPI_SWIGLU_BWD ? e.aux : e.resid;
            const void* pb = EPI == EPI_SWIGLU_BWD ? e.aux2 : e.aux;
            const int64_t ra = static_cast<int64_t>(m) * (EPI == EPI_SWIGLU_BWD ? e.ld_aux : e.ld_resid);
            const int64_t rb = static_cast<int64_t>(m) * (EPI == EPI_SWIGLU_BWD ? e.ld_aux2 : e.ld_aux);
            if (has_a) load_chunk_bf16(pa, ra, n0 + 32 * c0, p.N, xa, 0);
            if (has_b) load_chunk_bf16(pb, rb, n0 + 32 * c0, p.N, xb, 0);
            if (kb_total > 0) {
                if (!mbar_wait_bounded(&tfull[acc], (it >> 1) & 1, abort_flag)) break;
                tc_fence_after();
            }
            const uint32_t tbase = tmem_base + (static_cast<uint32_t>(q * 32) << 16) + static_cast<uint32_t>(acc * BN);
            float v[32];

            if constexpr (EPI == EPI_LINEAR) {
                const EpiRow r = epi_row(e, m, p.M);
                float t[32];
#pragma unroll 1
                for (int j = 0; j < CPW; ++j) {
                    const int c = c0 + j;
                    const int n = n0 + c * 32;
                    if (n >= p.N) break;
                    if (kb_total > 0) {
                        tmem_load32(tbase + c * 32, v);
                    } else {
#pragma unroll
                        for (int i = 0; i < 32; ++i) v[i] = 0.0f;
                    }
                    if (valid) {
#pragma unroll
                        for (int i = 0; i < 32; ++i) v[i] *= r.alpha;
                        if (e.bias) {
                            load_row32(e.bias, 0, n, p.N, 0, t);
#pragma unroll
                            for (int i = 0; i < 32; ++i) v[i] += t[i];
                        }
                        if (e.r1u) {
                            load_vec32(e.r1v, n, p.N, t);
#pragma unroll
                            for (int i = 0; i < 32; ++i) v[i] += r.beta_r1 * t[i];
                        }
                        if (e.bw) {
                            load_vec32(e.bw, n, p.N, t);
#pragma unroll
                            for (int i = 0; i < 32; ++i) v[i] += r.beta_bw * t[i];
                        }
                        if (has_a) {
                            unpack32_dyn(xa, 0, t);
                            if (j + 1 < CPW) load_chunk_bf16(pa, ra, n + 32, p.N, xa, 0);
#pragma unroll
                            for (int i = 0; i < 32; ++i) v[i] += t[i];
                        }
                        if (e.act == ACT_GELU) {
                            store_row32(e.out2, static_cast<int64_t>(m) * e.ld_out2, n, p.N, e.out2_f32, v);
#pragma unroll
                            for (int i = 0; i < 32; ++i) v[i] = gelu_f(e.out2_f32 ? v[i] : round_bf16(v[i]));
                        } else if (has_b) {
                            unpack32_dyn(xb, 0, t);
                            if (j + 1 < CPW) load_chunk_bf16(pb, rb, n + 32, p.N, xb, 0);
#pragma unroll
                            for (int i = 0; i < 32; ++i) v[i] *= gelu_grad_f(t[i]);
                        }
                        store_row32(e.out, static_cast<int64_t>(m) * e.ld_out, n, p.N, e.out_f32, v);
                    }
                }
            } else if constexpr (EPI == EPI_LOGITS) {
                // per (row, column half) softmax statistics: stats pair nt*2 + h
                float mx = -INFINITY, sm = 0.0f;
                float t[32];
#pragma unroll 1
                for (int j = 0; j < CPW; ++j) {
                    const int c = c0 + j;
                    const int n = n0 + c * 32;
                    if (n >= p.N) break;
                    tmem_load32(tbase + c * 32, v);
                    if (e.bias) {
                        load_row32(e.bias, 0, n, p.N, 0, t);
#pragma unroll
                        for (int i = 0; i < 32; ++i) v[i] += t[i];
                    }
                    if (!e.out_f32) {
#pragma unroll
                        for (int i = 0; i < 32; ++i) v[i] = round_bf16(v[i]);
                    }
                    if (valid) store_row32(e.out, static_cast<int64_t>(m) * e.ld_out, n, p.N, e.out_f32, v);
                    float cm = -INFINITY;
#pragma unroll
                    for (int i = 0; i < 32; ++i)
                        if (n + i < p.N) cm = fmaxf(cm, v[i]);
                    const float nm = fmaxf(mx, cm);
                    float s = (mx == -INFINITY) ? 0.0f : sm * fast_exp(mx - nm);
#pragma unroll
                    for (int i = 0; i < 32; ++i)
                        if (n + i < p.N) s += fast_exp(v[i] - nm);
                    mx = nm;
                    sm = s;
                }
                if (valid) {
                    float2* st = reinterpret_cast<float2*>(e.stats) + static_cast<int64_t>(m) * e.ld_stats + 2 * nt + h;
                    *st = make_float2(mx, sm);
                }
            } else if constexpr (EPI == EPI_SWIGLU_FWD) {
                // gate columns [0, 128) and up columns [128, 256) of the accumulator
                float u[32];
#pragma unroll 1
                for (int j = 0; j < 2; ++j) {
                    const int c = 2 * h + j;
                    const int n = n0 + c * 32;
                    if (n >= p.N) break;
                    tmem_load32(tbase + c * 32, v);
                    tmem_load32(tbase + 128 + c * 32, u);
                    if (valid) {
                        store_row32(e.out2, static_cast<int64_t>(m) * e.ld_out2, n, p.N, e.out2_f32, v);
                        store_row32(e.out3, static_cast<int64_t>(m) * e.ld_out3, n, p.N, e.out2_f32, u);
#pragma unroll
                        for (int i = 0; i < 32; ++i) {
                            const float g = round_bf16(v[i]);
                            v[i] = g * fast_sigmoid(g) * round_bf16(u[i]);
                        }
                        store_row32(e.out, static_cast<int64_t>(m) * e.ld_out, n, p.N, e.out_f32, v);
                    }
                }
            } else if constexpr (EPI == EPI_SWIGLU_BWD) {
                float g[32], u[32];
#pragma unroll 1
                for (int j = 0; j < CPW; ++j) {
                    const int c = c0 + j;
                    const int n = n0 + c * 32;
                    if (n >= p.N) break;
                    tmem_load32(tbase + c * 32, v);
                    if (valid) {
                        unpack32_dyn(xa, 0, g);
                        unpack32_dyn(xb, 0, u);
                        if (j + 1 < CPW) {
                            load_chunk_bf16(pa, ra, n + 32, p.N, xa, 0);
                            load_chunk_bf16(pb, rb, n + 32, p.N, xb, 0);
                        }
                        float du[32];
#pragma unroll
                        for (int i = 0; i < 32; ++i) {
                            const float sg = fast_sigmoid(g[i]);
                            du[i] = v[i] * g[i] * sg;
                            v[i] = v[i] * u[i] * sg * (1.0f + g[i] * (1.0f - sg));
                        }
                        store_row32(e.out, static_cast<int64_t>(m) * e.ld_out, n, p.N, e.out_f32, v);
                        store_row32(e.out2, static_cast<int64_t>(m) * e.ld_out2, n, p.N, e.out2_f32, du);
                    }
                }
            }
            tc_fence_before();
            mbar_arrive(&tempty[acc]);
        }
    }

    __syncthreads();
    if (warp == 1) {
        __syncwarp();
        tc_fence_after();
        tmem_dealloc(tmem_base, TMEM_COLS);
    }
    if (threadIdx.x == 0 && *abort_flag && p.epi.sc != nullptr)
        latch_status(const_cast<DevScalars*>(p.epi.sc), BOM_ETIMEOUT);
}

// ------------------------------------------------------------------ host side
static PFN_cuTensorMapEncodeTiled_v12000 encode_fn() {
    static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
    static std::once_flag once;
    std::call_once(once, [] {
        void* p = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
                cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
    });
    return fn;
}

// 2-D bf16 tensor map: `inner` contiguous elements per row, `outer` rows of
// pitch `ld` elements; box of box_inner x box_outer with 128-byte swizzle.
static bool make_map(CUtensorMap* map, const void* ptr, int64_t inner, int64_t outer, int64_t ld,
                     uint32_t box_inner, uint32_t box_outer) {
    auto fn = encode_fn();
    if (!fn) return false;
    if ((reinterpret_cast<uintptr_t>(ptr) & 15u) != 0) return false;
    if ((ld * 2) % 16 != 0 || inner < 1 || outer < 1 || ld < inner) return false;
    cuuint64_t dims[2] = {static_cast<cuuint64_t>(inner), static_cast<cuuint64_t>(outer)};
    cuuint64_t strides[1] = {static_cast<cuuint64_t>(ld * 2)};
    cuuint32_t box[2] = {box_inner, box_outer};
    cuuint32_t estr[2] = {1, 1};
    CUresult r = fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(ptr), dims, strides, box, estr,
                    CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                    CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    return r == CUDA_SUCCESS;
}

static bool map_operand(CUtensorMap* map, const Operand& o, int64_t rows, int64_t K, uint32_t rows_box) {
    if (o.mn_major) return make_map(map, o.ptr, rows, K, o.ld, 64, 64);
    return make_map(map, o.ptr, K, rows, o.ld, 64, rows_box);
}

template <bool A_MN, bool B_MN, int EPI>
static int launch_inst(const Params& p, int grid, cudaStream_t stream) {
    static bool attr_set = false;
    auto k = gemm_kernel<A_MN, B_MN, EPI>;
    if (!attr_set) {
        if (cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, SMEM_BYTES) != cudaSuccess)
            return BOM_ECUDA;
        attr_set = true;
    }
    k<<<grid, NUM_THREADS, SMEM_BYTES, stream>>>(p); count_launch();
    return cudaPeekAtLastError() == cudaSuccess ? BOM_OK : BOM_ECUDA;
}

}  // namespace tc

int device_sm_count() {
    static int n = 0;
    if (n == 0) {
        int dev = 0;
        cudaGetDevice(&dev);
        cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev);
        if (n <= 0) n = 1;
    }
    return n;
}

int64_t tc_logit_tiles(int64_t N) { return 2 * ((N + tc::BN - 1) / tc::BN); }  // one pair per column half

int launch_gemm_tc(const GemmDesc& g, cudaStream_t stream) {
    using namespace tc;
    if (g.M <= 0 || g.N <= 0) return BOM_OK;
    if (g.M > INT32_MAX / 2 || g.N > INT32_MAX / 2) return BOM_ENOTSUP;
    if (g.epi.in_f32) return BOM_ENOTSUP;   // epilogue operands are bf16 on this engine
    Params p;
    memset(&p, 0, sizeof(p));
    const bool a_mn = g.A[0].mn_major, b_mn = g.B[0].mn_major;
    for (int s = 0; s < g.nseg; ++s) {
        if (g.A[s].mn_major != a_mn || g.B[s].mn_major != b_mn) return BOM_ENOTSUP;
        p.kb[s] = static_cast<int>((g.K[s] + BK - 1) / BK);
        if (g.K[s] <= 0) continue;
        if (!map_operand(&p.mapA[s], g.A[s], g.M, g.K[s], BM)) return BOM_ENOTSUP;
        if (g.dual_b) {
            if (b_mn || g.nseg != 1) return BOM_ENOTSUP;
            if (!map_operand(&p.mapB[0], g.B[0], g.N, g.K[0], 128)) return BOM_ENOTSUP;
            if (!map_operand(&p.mapB[1], g.B[1], g.N, g.K[0], 128)) return BOM_ENOTSUP;
        } else if (!map_operand(&p.mapB[s], g.B[s], g.N, g.K[s], BN)) {
            return BOM_ENOTSUP;
        }
    }
    p.M = static_cast<int>(g.M);
    p.N = static_cast<int>(g.N);
    p.nseg = g.nseg;
    p.dual_b = g.dual_b ? 1 : 0;
    p.bn_out = g.dual_b ? 128 : BN;
    p.tiles_m = static_cast<int>((g.M + BM - 1) / BM);
    p.tiles_n = static_cast<int>((g.N + p.bn_out - 1) / p.bn_out);
    p.epi = g.epi;
    const int tiles = p.tiles_m * p.tiles_n;
    const int grid = tiles < device_sm_count() ? tiles : device_sm_count();

    switch (g.epi_kind) {
        case EPI_LINEAR:
            if (!a_mn && !b_mn) return launch_inst<false, false, EPI_LINEAR>(p, grid, stream);
            if (!a_mn && b_mn) return launch_inst<false, true, EPI_LINEAR>(p, grid, stream);
            if (a_mn && b_mn) return launch_inst<true, true, EPI_LINEAR>(p, grid, stream);
            return launch_inst<true, false, EPI_LINEAR>(p, grid, stream);
        case EPI_LOGITS:
            if (a_mn || b_mn) return BOM_ENOTSUP;
            return launch_inst<false, false, EPI_LOGITS>(p, grid, stream);
        case EPI_SWIGLU_FWD:
            if (a_mn || !g.dual_b) return BOM_ENOTSUP;
            return launch_inst<false, false, EPI_SWIGLU_FWD>(p, grid, stream);
        case EPI_SWIGLU_BWD:
            if (a_mn || !b_mn) return BOM_ENOTSUP;
            return launch_inst<false, true, EPI_SWIGLU_BWD>(p, grid, stream);
        default:
            return BOM_EINVAL;
    }
}

}  // namespace bom
