// tcgen05 GEMM engine for sm_103a: bf16 operands, fp32 accumulation in TMEM.
//
// Persistent kernel.  When M > 128, CTA pairs (clusters of two, one pair per
// two SMs) compute 256 x 256 output tiles with cta_group::2 UMMAs; otherwise
// single CTAs compute 128 x 256 tiles (128 x 128 output columns when the B
// tile is split between gate and up weights).  Warp roles:
//   warp 0     one thread issues TMA tile loads (128-byte swizzle) into a
//              shared-memory ring guarded by mbarriers: as many stages (A
//              rows and this CTA's part of B: 32 KB for a CTA pair) as fit,
//              at most six;
//   warp 1     allocates 512 TMEM columns (two 256-column fp32 accumulators)
//              and, in the even CTA, one thread issues the UMMAs (K = 16),
//              releasing each smem stage with tcgen05.commit;
//   warps 2-9  epilogue: tcgen05.ld of the accumulator (one TMEM lane = one
//              output row per thread; two warps per lane quarter, one per
//              column half), the fused epilogue of the step, and global
//              stores.  With two accumulators the epilogue of tile i overlaps
//              the mainloop of tile i+1.
// Every mbarrier wait is bounded; a wait that runs out latches BOM_ETIMEOUT,
// all roles unwind, in-flight TMA loads and UMMAs are drained, TMEM is freed.
#include <atomic>
#include <cmath>
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
constexpr int NUM_THREADS = 320;  // producer warp, UMMA warp, 8 epilogue warps
// Narrow single-CTA tiles (128 x 64) for linear-epilogue GEMMs whose 256 x 256
// tiles would keep at most a quarter of the SMs busy: the epilogue of such a
// GEMM (bias, GELU or its derivative, residual, one row per thread) takes
// longer than its mainloop, and 128 x 64 tiles spread it over four times as
// many SMs.
constexpr int kBnSmall = 64;
// Tile raster: groups of group_m consecutive m-tiles with m fastest inside a
// group (group_m = 1: n fastest along whole rows of tiles).  See raster_group.
constexpr int GROUP_M = 8;

constexpr int kMaxGroup = 8;
struct Prob {
    CUtensorMap mapA, mapB;
    int M, N, tiles_m, tiles_n, group_m;
    EpiParams epi;
};

struct Params {
    CUtensorMap mapA[2];
    CUtensorMap mapB[2];
    int M, N;
    int kb[2];
    int nseg;
    int tiles_m, tiles_n;
    int group_m;           // raster group of problem 0 (raster_group)
    int dual_b;
    int bn_out;
    int ksplit;            // K ranges per output tile (1: no split)
    int kb_split;          // k-blocks per K range
    int64_t split_bytes;   // byte distance between the fp32 partial slices of e.out
    EpiParams epi;
    // Grouped launch: problems 1.. of the group (problem 0 is the fields
    // above).  All problems share the layout, the epilogue kind and K; their
    // tiles are numbered one problem after the other.
    int nprob;
    int tile_base[kMaxGroup + 1];
    Prob grp[kMaxGroup - 1];
};

static_assert(sizeof(Params) <= 32764, "kernel parameters exceed the launch limit");

// Problem of `tile` (a tile index over the whole group) and its tile within it.
struct ProbView {
    const CUtensorMap* mapA;
    const CUtensorMap* mapB;
    const EpiParams* epi;
    int M, N, tiles_m, tiles_n, group_m, local;
};
__device__ __forceinline__ ProbView prob_of(const Params& p, int tile) {
    int q = 0;
    while (q + 1 < p.nprob && tile >= p.tile_base[q + 1]) ++q;
    ProbView v;
    if (q == 0) {
        v.mapA = &p.mapA[0];
        v.mapB = &p.mapB[0];
        v.epi = &p.epi;
        v.M = p.M;
        v.N = p.N;
        v.tiles_m = p.tiles_m;
        v.tiles_n = p.tiles_n;
        v.group_m = p.group_m;
    } else {
        const Prob& g = p.grp[q - 1];
        v.mapA = &g.mapA;
        v.mapB = &g.mapB;
        v.epi = &g.epi;
        v.M = g.M;
        v.N = g.N;
        v.tiles_m = g.tiles_m;
        v.tiles_n = g.tiles_n;
        v.group_m = g.group_m;
    }
    v.local = tile - p.tile_base[q];
    return v;
}

__device__ __forceinline__ void tile_coords(int tile, int tiles_m, int tiles_n, int group_m, int& mt, int& nt) {
    const int per_group = group_m * tiles_n;
    const int g = tile / per_group;
    const int first_m = g * group_m;
    const int gsz = min(tiles_m - first_m, group_m);
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
    if (n + 32 <= N && (reinterpret_cast<uintptr_t>(p) & 31u) == 0) {
        // two whole 32-byte sectors in 256-bit loads
#pragma unroll
        for (int i = 0; i < 2; ++i) {
            uint4 a, b;
            asm("ld.global.nc.v8.b32 {%0, %1, %2, %3, %4, %5, %6, %7}, [%8];"
                         : "=r"(a.x), "=r"(a.y), "=r"(a.z), "=r"(a.w), "=r"(b.x), "=r"(b.y), "=r"(b.z), "=r"(b.w)
                         : "l"(p + 16 * i));
            pk[4 * slot + 2 * i] = a;
            pk[4 * slot + 2 * i + 1] = b;
        }
    } else if (n + 32 <= N) {
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

// 32 bytes from a 32-byte aligned global address in one 256-bit load (plain,
// coherent: the fused update rewrites what it reads).
__device__ __forceinline__ void ld_global_v8(const void* p, float (&v)[8]) {
    uint32_t r[8];
    asm volatile("ld.global.v8.b32 {%0, %1, %2, %3, %4, %5, %6, %7}, [%8];"
                 : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7])
                 : "l"(p)
                 : "memory");
#pragma unroll
    for (int i = 0; i < 8; ++i) v[i] = __uint_as_float(r[i]);
}

// BOM-AdamW update of one element (Section 3.4): v' = b2 v + (1-b2) u^2,
// theta' = (1 - lr wd) theta - lr u / (sqrt(v' / (1-b2^t)) + eps), with the
// hardware square root and reciprocal.
__device__ __forceinline__ void update1(const EpiParams& e, float u, float& th, float& v, float lr, float decay,
                                        float inv_bc2) {
    v = fmaf(e.upd_beta2, v, e.upd_1mb2 * u * u);
    th = apply_step(decay, th, lr, u * rcp_fast(sqrt_fast(v * inv_bc2) + e.upd_eps));
}

// Fused update, one row per lane: lane l holds u of its own row m, columns
// [n, n + 32), and reads and rewrites that row's theta and v and writes its
// compute copy.  Where the row segment is whole and 32-byte aligned every
// access is a 256-bit load or store of a whole sector (16 columns of theta and
// v in flight at a time), as in the other epilogues; 16-byte aligned rows take
// 128-bit accesses, ragged ones single elements.  Against a transpose of
// each 32 x 32 block through shared memory (to walk theta and v in 128-byte
// lines by rows) it issues about a ninth as many memory instructions for the
// same sectors, and the grouped weight-gradient launch of the LM block took
// 3.24 instead of 3.33 ms (same-box A/B).
__device__ __forceinline__ void row_update32(const EpiParams& e, int m, int M, int n, int N, const float (&u)[32],
                                             float lr, float decay, float inv_bc2) {
    if (m >= M) return;
    const int64_t off = static_cast<int64_t>(m) * e.ld_out + n;
    float* const th = e.upd_theta + off;
    float* const vv = e.upd_v + off;
    float t2[32];
    if (n + 32 <= N && ((reinterpret_cast<uintptr_t>(th) | reinterpret_cast<uintptr_t>(vv)) & 31u) == 0) {
#pragma unroll
        for (int h = 0; h < 2; ++h) {
            float a[2][8], b[2][8];
#pragma unroll
            for (int k = 0; k < 2; ++k) {
                ld_global_v8(th + 16 * h + 8 * k, a[k]);
                ld_global_v8(vv + 16 * h + 8 * k, b[k]);
            }
#pragma unroll
            for (int k = 0; k < 2; ++k) {
#pragma unroll
                for (int i = 0; i < 8; ++i) {
                    update1(e, u[16 * h + 8 * k + i], a[k][i], b[k][i], lr, decay, inv_bc2);
                    t2[16 * h + 8 * k + i] = a[k][i];
                }
                st_global_v8(th + 16 * h + 8 * k, __float_as_uint(a[k][0]), __float_as_uint(a[k][1]),
                             __float_as_uint(a[k][2]), __float_as_uint(a[k][3]), __float_as_uint(a[k][4]),
                             __float_as_uint(a[k][5]), __float_as_uint(a[k][6]), __float_as_uint(a[k][7]));
                st_global_v8(vv + 16 * h + 8 * k, __float_as_uint(b[k][0]), __float_as_uint(b[k][1]),
                             __float_as_uint(b[k][2]), __float_as_uint(b[k][3]), __float_as_uint(b[k][4]),
                             __float_as_uint(b[k][5]), __float_as_uint(b[k][6]), __float_as_uint(b[k][7]));
            }
        }
    } else if (n + 32 <= N && ((reinterpret_cast<uintptr_t>(th) | reinterpret_cast<uintptr_t>(vv)) & 15u) == 0) {
        // rows that are only 16-byte aligned: 128-bit accesses, 8 columns at a time
#pragma unroll
        for (int k = 0; k < 4; ++k) {
            float4 a[2], b[2];
#pragma unroll
            for (int j = 0; j < 2; ++j) {
                a[j] = reinterpret_cast<const float4*>(th)[2 * k + j];
                b[j] = reinterpret_cast<const float4*>(vv)[2 * k + j];
            }
#pragma unroll
            for (int j = 0; j < 2; ++j) {
                float* pa = &a[j].x;
                float* pb = &b[j].x;
#pragma unroll
                for (int i = 0; i < 4; ++i) {
                    update1(e, u[8 * k + 4 * j + i], pa[i], pb[i], lr, decay, inv_bc2);
                    t2[8 * k + 4 * j + i] = pa[i];
                }
                reinterpret_cast<float4*>(th)[2 * k + j] = a[j];
                reinterpret_cast<float4*>(vv)[2 * k + j] = b[j];
            }
        }
    } else {
#pragma unroll
        for (int i = 0; i < 32; ++i) {
            t2[i] = 0.0f;
            if (n + i < N) {
                float a = th[i], b = vv[i];
                update1(e, u[i], a, b, lr, decay, inv_bc2);
                th[i] = a;
                vv[i] = b;
                t2[i] = a;
            }
        }
    }
    store_row32(e.out, static_cast<int64_t>(m) * e.ld_out, n, N, e.out_f32, t2);
}

__device__ __forceinline__ float fast_exp(float x) { return exp2f(x * 1.4426950408889634f); }

__device__ __forceinline__ void tmem_load32(uint32_t taddr, float (&v)[32]) {
    uint32_t r[32];
    __syncwarp();
    tmem_ld_32x32b_x32(taddr, r);
    tmem_ld_wait();
#pragma unroll
    for (int i = 0; i < 32; ++i) v[i] = __uint_as_float(r[i]);
}

// Shared-memory layout of one CTA.  CG = 1: the CTA computes 128 x 256 tiles
// alone.  CG = 2: a CTA pair (cluster of 2) computes 256 x 256 tiles with
// tcgen05 cta_group::2 UMMAs issued by the even CTA; each CTA stages its own
// 128 rows of A and its half (128 rows) of B, so a stage is 32 KB.  Epilogue
// stores go straight from each lane's row to global memory in 256-bit stores
// (whole 32-byte sectors); staging them through shared memory cost pipeline
// stages and measured slower.  The fused update reads and rewrites theta and v
// the same way, one row per lane.
// SwiGLU backward: the epilogue's per-row operands (the saved G and U,
// interleaved per 32 columns in one 128-byte line of a row) are read by each
// lane for its own row in four 256-bit loads, the next chunk's line while the
// current one is processed.

// One 128-byte line (a [G 32 | U 32] block of the interleaved saved gate and up
// pre-activations, 32-byte aligned) in four 256-bit loads: G in w[0..3], U in w[4..7].
__device__ __forceinline__ void load_line128(const void* p, uint4 (&w)[8]) {
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        uint4 a, b;
        asm("ld.global.nc.v8.b32 {%0, %1, %2, %3, %4, %5, %6, %7}, [%8];"
            : "=r"(a.x), "=r"(a.y), "=r"(a.z), "=r"(a.w), "=r"(b.x), "=r"(b.y), "=r"(b.z), "=r"(b.w)
            : "l"(static_cast<const char*>(p) + 32 * i));
        w[2 * i] = a;
        w[2 * i + 1] = b;
    }
}

template <int CG, int EPI, int BNT>
struct Cfg {
    static_assert(BNT == BN || (CG == 1 && BNT == kBnSmall), "narrow tiles are single-CTA only");
    static constexpr int B_ROWS = CG == 2 ? BN / 2 : BNT;
    // two accumulators of BNT fp32 columns (an allocation is a power of two >= 32)
    static constexpr int TMEM_COLS = 2 * BNT;
    static constexpr int A_BYTES = BM * BK * 2;
    static constexpr int B_BYTES = B_ROWS * BK * 2;
    static constexpr int BAR_BYTES = 512;
    // as many stages as fit in the 227 KB a CTA may use beside the 1 KB
    // alignment slack and the barrier block, at most six (a seventh 32 KB
    // stage measured slower on the linear and SwiGLU backward epilogues, and
    // no faster under the fused update)
    static constexpr int STAGES_FIT = (227 * 1024 - 1024 - BAR_BYTES) / (A_BYTES + B_BYTES);
    static constexpr int STAGES = STAGES_FIT < 6 ? STAGES_FIT : 6;
    static constexpr int SMEM = STAGES * (A_BYTES + B_BYTES) + 1024 + BAR_BYTES;
    static_assert(STAGES >= 2, "pipeline needs two stages");
    static constexpr int TILE_M = BM * CG;
};

template <int CG, bool A_MN, bool B_MN, int EPI, int BNT>
__global__ void __launch_bounds__(NUM_THREADS, 1) gemm_kernel(const __grid_constant__ Params p) {
    // the next kernel may be scheduled now; this one's own set-up (barriers,
    // TMEM, tensor-map prefetch) runs before it waits for the previous kernel
    pdl_trigger();
    using C = Cfg<CG, EPI, BNT>;
    constexpr int STAGES = C::STAGES;
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    uint8_t* sA = smem;
    uint8_t* sB = smem + STAGES * C::A_BYTES;
    uint64_t* bars = reinterpret_cast<uint64_t*>(sB + STAGES * C::B_BYTES);
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
    const uint32_t rank = CG == 2 ? cluster_ctarank() : 0u;
    const bool leader = rank == 0;
    const int unit = CG == 2 ? static_cast<int>(blockIdx.x >> 1) : static_cast<int>(blockIdx.x);
    const int nunits = CG == 2 ? static_cast<int>(gridDim.x >> 1) : static_cast<int>(gridDim.x);

    if (threadIdx.x == 0) {
        for (int s = 0; s < STAGES; ++s) {
            mbar_init(&full[s], 1);
            mbar_init(&empty[s], 1);
        }
        for (int a = 0; a < 2; ++a) {
            mbar_init(&tfull[a], 1);
            // CG = 2: one elected arrival per CTA of the pair on the even CTA's barrier
            mbar_init(&tempty[a], CG == 2 ? 2 : 256);
        }
        mbar_init(drain, 1);
        *abort_flag = 0;
        fence_barrier_init();
    }
    if (warp == 0 && lane == 0) {
        prefetch_tensormap(&p.mapA[0]);
        prefetch_tensormap(&p.mapB[0]);
    }
    if (warp == 1) {
        if constexpr (CG == 2) {
            tmem_alloc_pair(tmem_slot, C::TMEM_COLS);
            tmem_relinquish_pair();
        } else {
            tmem_alloc(tmem_slot, C::TMEM_COLS);
            tmem_relinquish();
        }
    }
    tc_fence_before();
    __syncthreads();
    if constexpr (CG == 2) cluster_sync();   // barriers of both CTAs initialised before any remote use
    tc_fence_after();
    pdl_wait();   // the previous kernel's writes (operands, status word) are visible from here on
    if (threadIdx.x == 0) *skip_flag = (p.epi.sc != nullptr && p.epi.sc->status != 0) ? 1 : 0;
    __syncthreads();
    const uint32_t tmem_base = *tmem_slot;
    const bool skip = *skip_flag != 0;

    const int num_tiles = p.tile_base[p.nprob];
    const int num_work = num_tiles * p.ksplit;   // (tile, K-split) work units
    const int kb_total = p.kb[0] + (p.nseg > 1 ? p.kb[1] : 0);

    if (!skip && warp == 0) {
        // ------------------------------------------------------------ TMA producer
        if (lane == 0 && kb_total > 0) {
            int stage = 0;
            uint32_t phase = 0;
            uint32_t issued_mask = 0, issued_phase = 0;
            bool ok = true;
            for (int w = unit; ok && w < num_work; w += nunits) {
                const int tile = w / p.ksplit;
                const int sp = w - tile * p.ksplit;
                const ProbView pv = prob_of(p, tile);
                int mt, nt;
                tile_coords(pv.local, pv.tiles_m, pv.tiles_n, pv.group_m, mt, nt);
                const int m_own = mt * C::TILE_M + static_cast<int>(rank) * BM;
                const int n0 = nt * p.bn_out;
                const int n_own = n0 + (CG == 2 && !p.dual_b ? static_cast<int>(rank) * C::B_ROWS : 0);
                const int g0 = sp * p.kb_split;
                const int g1 = min(g0 + p.kb_split, kb_total);
                {
                    for (int gk = g0; gk < g1; ++gk) {
                        const int seg = gk < p.kb[0] ? 0 : 1;
                        const int kb = seg == 0 ? gk : gk - p.kb[0];
                        if (!mbar_wait_bounded(&empty[stage], phase ^ 1u, abort_flag)) {
                            ok = false;
                            break;
                        }
                        if (leader) mbar_arrive_expect_tx(&full[stage], CG * (C::A_BYTES + C::B_BYTES));
                        const int k0 = kb * BK;
                        uint8_t* a = sA + stage * C::A_BYTES;
                        uint8_t* b = sB + stage * C::B_BYTES;
                        auto load = [&](void* dst, const CUtensorMap* map, int x, int y) {
                            if constexpr (CG == 2)
                                tma_load_2d_pair(dst, map, mapa_shared(smem_u32(&full[stage]), 0), x, y);
                            else
                                tma_load_2d(dst, map, &full[stage], x, y);
                        };
                        // grouped problems have one K segment: their maps come from pv
                        const CUtensorMap* mA = seg == 0 ? pv.mapA : &p.mapA[1];
                        const CUtensorMap* mB = seg == 0 ? pv.mapB : &p.mapB[1];
                        if (!A_MN) {
                            load(a, mA, k0, m_own);
                        } else {
                            load(a, mA, m_own, k0);
                            load(a + 8192, mA, m_own + 64, k0);
                        }
                        if (p.dual_b) {
                            if constexpr (CG == 2) {
                                load(b, &p.mapB[rank], k0, n0);   // even CTA: gate rows, odd CTA: up rows
                            } else {
                                load(b, &p.mapB[0], k0, n0);
                                load(b + 16384, &p.mapB[1], k0, n0);
                            }
                        } else if (!B_MN) {
                            load(b, mB, k0, n_own);
                        } else {
#pragma unroll
                            for (int j = 0; j < C::B_ROWS / 64; ++j) load(b + j * 8192, mB, n_own + 64 * j, k0);
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
            // Every issued load must land before the CTA may exit (the even CTA's
            // full barriers also count the odd CTA's loads).
            if (leader)
                for (int s = 0; s < STAGES; ++s)
                    if (issued_mask & (1u << s)) mbar_wait_bounded(&full[s], (issued_phase >> s) & 1u, nullptr);
        }
    } else if (!skip && warp == 1) {
        // ------------------------------------------------------------ UMMA issuer (even CTA)
        if (lane == 0 && kb_total > 0 && leader) {
            constexpr uint32_t idesc = idesc_bf16_f32(C::TILE_M, BNT, A_MN, B_MN);
            constexpr uint32_t b_lbo = 8192;   // MN-major: next 64-column chunk
            int stage = 0;
            uint32_t phase = 0;
            bool ok = true;
            int it = 0;
            for (int w = unit; ok && w < num_work; w += nunits, ++it) {
                const int acc = it & 1;
                const uint32_t aph = (it >> 1) & 1;
                const int sp = w % p.ksplit;
                const int nk = min(p.kb_split, kb_total - sp * p.kb_split);
                if (!mbar_wait_bounded(&tempty[acc], aph ^ 1u, abort_flag)) break;
                tc_fence_after();
                const uint32_t d_tmem = tmem_base + static_cast<uint32_t>(acc * BNT);
                for (int kb = 0; kb < nk; ++kb) {
                    if (!mbar_wait_bounded(&full[stage], phase, abort_flag)) {
                        ok = false;
                        break;
                    }
                    tc_fence_after();
                    const uint32_t a0 = smem_u32(sA + stage * C::A_BYTES);
                    const uint32_t b0 = smem_u32(sB + stage * C::B_BYTES);
#pragma unroll
                    for (int kk = 0; kk < BK / 16; ++kk) {
                        const uint64_t ad = A_MN ? smem_desc_sw128(a0 + kk * 2048, 8192, 1024)
                                                 : smem_desc_sw128(a0 + kk * 32, 16, 1024);
                        const uint64_t bd = B_MN ? smem_desc_sw128(b0 + kk * 2048, b_lbo, 1024)
                                                 : smem_desc_sw128(b0 + kk * 32, 16, 1024);
                        if constexpr (CG == 2)
                            umma_bf16_pair(d_tmem, ad, bd, idesc, (kb | kk) != 0 ? 1u : 0u);
                        else
                            umma_bf16(d_tmem, ad, bd, idesc, (kb | kk) != 0 ? 1u : 0u);
                    }
                    if constexpr (CG == 2)
                        umma_commit_pair(&empty[stage], 0x3);
                    else
                        umma_commit(&empty[stage]);
                    if (++stage == STAGES) {
                        stage = 0;
                        phase ^= 1u;
                    }
                }
                if (ok) {
                    if constexpr (CG == 2)
                        umma_commit_pair(&tfull[acc], 0x3);
                    else
                        umma_commit(&tfull[acc]);
                }
            }
            // All issued UMMAs must finish before TMEM is released.
            if constexpr (CG == 2)
                umma_commit_pair(drain, 0x1);
            else
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
        constexpr int CPW = BNT / 64;  // 32-column chunks per warp
        int it = 0;
        for (int w = unit; w < num_work; w += nunits, ++it) {
            const int tile = w / p.ksplit;
            const ProbView pv = prob_of(p, tile);
            const EpiParams& e = *pv.epi;
            const int PM = pv.M, PN = pv.N;
            // split-K: each K range stores its raw fp32 tile into its own slice
            void* const out_base = static_cast<char*>(e.out) + static_cast<int64_t>(w - tile * p.ksplit) * p.split_bytes;
            int mt, nt;
            tile_coords(pv.local, pv.tiles_m, pv.tiles_n, pv.group_m, mt, nt);
            const int m0 = mt * C::TILE_M + static_cast<int>(rank) * BM;
            const int n0 = nt * p.bn_out;
            const int acc = it & 1;
            const int m = m0 + row;
            const bool valid = m < PM;
            const int c0 = h * CPW;
            // Per-row epilogue operands do not depend on the accumulator: the
            // warp's first chunk is loaded before the mainloop wait, and each
            // later chunk while the previous one is being processed.
            uint4 xa[4], xb[4];
            uint4 gu[8];   // SwiGLU backward: the current chunk's [G 32 | U 32] line
            const bool has_a = valid && ((EPI == EPI_SWIGLU_BWD) || (EPI == EPI_LINEAR && e.resid != nullptr));
            const bool has_b = valid && ((EPI == EPI_SWIGLU_BWD) || (EPI == EPI_LINEAR && e.act == ACT_DGELU));
            const void* pa = EPI == EPI_SWIGLU_BWD ? e.aux : e.resid;
            const void* pb = EPI == EPI_SWIGLU_BWD ? e.aux2 : e.aux;
            const int64_t ra = static_cast<int64_t>(m) * (EPI == EPI_SWIGLU_BWD ? e.ld_aux : e.ld_resid);
            const int64_t rb = static_cast<int64_t>(m) * (EPI == EPI_SWIGLU_BWD ? e.ld_aux2 : e.ld_aux);
            const int row0 = m0 + q * 32;   // first of the warp's 32 rows
            if (EPI == EPI_SWIGLU_BWD) {
                // the line of this warp's first chunk
                if (valid && n0 + 32 * c0 < PN)
                    load_line128(static_cast<const uint16_t*>(pa) + ra + 2 * (n0 + 32 * c0), gu);
            } else {
                if (has_a) load_chunk_bf16(pa, ra, n0 + 32 * c0, PN, xa, 0);
                if (has_b) load_chunk_bf16(pb, rb, n0 + 32 * c0, PN, xb, 0);
            }
            // linear epilogue: the row's factors, and on narrow tiles (one
            // chunk per warp) the chunk's bias and broadcast row, are read
            // before the accumulator is waited for
            EpiRow r_lin{};
            float vb[32], vw[32];
            if constexpr (EPI == EPI_LINEAR) {
                r_lin = epi_row(e, m, PM);
                if constexpr (CPW == 1) {
                    const int nf = n0 + 32 * c0;
                    if (valid && nf < PN) {
                        if (e.bias) load_row32(e.bias, 0, nf, PN, 0, vb);
                        if (e.bw) load_vec32(e.bw, nf, PN, vw);
                    }
                }
            }
            if (kb_total > 0) {
                if (!mbar_wait_bounded(&tfull[acc], (it >> 1) & 1, abort_flag)) break;
                tc_fence_after();
            }
            const uint32_t tbase = tmem_base + (static_cast<uint32_t>(q * 32) << 16) + static_cast<uint32_t>(acc * BNT);
            float v[32];

            if constexpr (EPI == EPI_LINEAR) {
                const EpiRow r = r_lin;
                float t[32];
#pragma unroll 1
                for (int j = 0; j < CPW; ++j) {
                    const int c = c0 + j;
                    const int n = n0 + c * 32;
                    if (n >= PN) break;
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
                            if (CPW > 1) load_row32(e.bias, 0, n, PN, 0, vb);
#pragma unroll
                            for (int i = 0; i < 32; ++i) v[i] += vb[i];
                        }
                        if (e.r1u) {
                            load_vec32(e.r1v, n, PN, t);
#pragma unroll
                            for (int i = 0; i < 32; ++i) v[i] += r.beta_r1 * t[i];
                        }
                        if (e.bw) {
                            if (CPW > 1) load_vec32(e.bw, n, PN, vw);
#pragma unroll
                            for (int i = 0; i < 32; ++i) v[i] += r.beta_bw * vw[i];
                        }
                        if (has_a) {
                            unpack32_dyn(xa, 0, t);
                            if (j + 1 < CPW) load_chunk_bf16(pa, ra, n + 32, PN, xa, 0);
#pragma unroll
                            for (int i = 0; i < 32; ++i) v[i] += t[i];
                        }
                        if (e.act == ACT_GELU) {
                            store_row32(e.out2, static_cast<int64_t>(m) * e.ld_out2, n, PN, e.out2_f32, v);
#pragma unroll
                            for (int i = 0; i < 32; ++i) v[i] = gelu_f(e.out2_f32 ? v[i] : round_bf16(v[i]));
                        } else if (has_b) {
                            unpack32_dyn(xb, 0, t);
                            if (j + 1 < CPW) load_chunk_bf16(pb, rb, n + 32, PN, xb, 0);
#pragma unroll
                            for (int i = 0; i < 32; ++i) v[i] *= gelu_grad_f(t[i]);
                        }
                        store_row32(out_base, static_cast<int64_t>(m) * e.ld_out, n, PN, e.out_f32, v);
                    }
                    if (e.colsum != nullptr) {
                        // the 32 rows of this warp, column by column: lane i
                        // ends with the sum of column n + i
#pragma unroll
                        for (int i = 0; i < 32; ++i) v[i] = valid ? (e.out_f32 ? v[i] : round_bf16(v[i])) : 0.0f;
                        const float cs = warp_colsum32(v, lane);
                        if (row0 < PM && n + lane < PN)
                            e.colsum[static_cast<int64_t>(row0 >> 5) * e.ld_colsum + n + lane] = cs;
                    }
                }
            } else if constexpr (EPI == EPI_UPDATE) {
                const EpiRow r = epi_row(e, m, PM);
                const float lr = e.sc->lr, inv_bc2 = e.sc->inv_bc2;
                const float decay = decay_factor(lr, e.upd_wd);
                float t[32];
#pragma unroll 1
                for (int j = 0; j < CPW; ++j) {
                    const int c = c0 + j;
                    const int n = n0 + c * 32;
                    if (n >= PN) break;
                    if (kb_total > 0) {
                        tmem_load32(tbase + c * 32, v);
                    } else {
#pragma unroll
                        for (int i = 0; i < 32; ++i) v[i] = 0.0f;
                    }
#pragma unroll
                    for (int i = 0; i < 32; ++i) v[i] *= r.alpha;
                    if (e.r1u) {
                        load_vec32(e.r1v, n, PN, t);
#pragma unroll
                        for (int i = 0; i < 32; ++i) v[i] += r.beta_r1 * t[i];
                    }
                    row_update32(e, m, PM, n, PN, v, lr, decay, inv_bc2);
                }
            } else if constexpr (EPI == EPI_LOGITS) {
                // per (row, column half) softmax statistics: stats pair nt*2 + h.
                // The statistics are taken over the bf16-rounded logits that
                // are stored, so the residual pass sees a consistent row.
                float mx = -INFINITY, sm = 0.0f;
                float t[32];
#pragma unroll 1
                for (int j = 0; j < CPW; ++j) {
                    const int c = c0 + j;
                    const int n = n0 + c * 32;
                    if (n >= PN) break;
                    tmem_load32(tbase + c * 32, v);
                    if (e.bias) {
                        load_row32(e.bias, 0, n, PN, 0, t);
#pragma unroll
                        for (int i = 0; i < 32; ++i) v[i] += t[i];
                    }
                    if (n + 32 <= PN) {
                        // full chunk: packed rounding, packed max, paired exponentials
                        uint32_t b[16];
#pragma unroll
                        for (int i = 0; i < 16; ++i) b[i] = cvt_bf16x2(v[2 * i], v[2 * i + 1]);
                        if (valid) {
                            uint16_t* dst16 = static_cast<uint16_t*>(e.out) + static_cast<int64_t>(m) * e.ld_out + n;
                            if ((reinterpret_cast<uintptr_t>(dst16) & 31u) == 0) {   // two whole-sector stores
                                st_global_v8(dst16, b[0], b[1], b[2], b[3], b[4], b[5], b[6], b[7]);
                                st_global_v8(dst16 + 16, b[8], b[9], b[10], b[11], b[12], b[13], b[14], b[15]);
                            } else {
                                uint4* dst = reinterpret_cast<uint4*>(dst16);
#pragma unroll
                                for (int i = 0; i < 4; ++i)
                                    dst[i] = make_uint4(b[4 * i], b[4 * i + 1], b[4 * i + 2], b[4 * i + 3]);
                            }
                        }
                        uint32_t mb[8];
#pragma unroll
                        for (int i = 0; i < 8; ++i) mb[i] = max_bf16x2(b[2 * i], b[2 * i + 1]);
#pragma unroll
                        for (int i = 0; i < 4; ++i) mb[i] = max_bf16x2(mb[i], mb[i + 4]);
                        mb[0] = max_bf16x2(max_bf16x2(mb[0], mb[2]), max_bf16x2(mb[1], mb[3]));
                        const float nm = fmaxf(mx, fmaxf(bf16_lo(mb[0]), bf16_hi(mb[0])));
                        const float2 l2 = make_float2(kLog2e, kLog2e);
                        const float2 off = make_float2(-nm * kLog2e, -nm * kLog2e);
                        float2 a0 = make_float2(0.0f, 0.0f), a1 = a0;
#pragma unroll
                        for (int i = 0; i < 16; i += 2) {
                            const float2 x0 = fma2(make_float2(bf16_lo(b[i]), bf16_hi(b[i])), l2, off);
                            const float2 x1 = fma2(make_float2(bf16_lo(b[i + 1]), bf16_hi(b[i + 1])), l2, off);
                            a0 = add2(a0, make_float2(ex2_fast(x0.x), ex2_fast(x0.y)));
                            a1 = add2(a1, make_float2(ex2_fast(x1.x), ex2_fast(x1.y)));
                        }
                        a0 = add2(a0, a1);
                        const float scale = (mx == -INFINITY) ? 0.0f : ex2_fast((mx - nm) * kLog2e);
                        sm = sm * scale + (a0.x + a0.y);
                        mx = nm;
                        continue;
                    }
                    // ragged last chunk
#pragma unroll
                    for (int i = 0; i < 32; ++i) v[i] = round_bf16(v[i]);
                    if (valid) store_row32(e.out, static_cast<int64_t>(m) * e.ld_out, n, PN, 0, v);
                    float cm = -INFINITY;
#pragma unroll
                    for (int i = 0; i < 32; ++i)
                        if (n + i < PN) cm = fmaxf(cm, v[i]);
                    const float nm = fmaxf(mx, cm);
                    float s = (mx == -INFINITY) ? 0.0f : sm * fast_exp(mx - nm);
#pragma unroll
                    for (int i = 0; i < 32; ++i)
                        if (n + i < PN) s += fast_exp(v[i] - nm);
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
                    if (n >= PN) break;
                    tmem_load32(tbase + c * 32, v);
                    tmem_load32(tbase + 128 + c * 32, u);
                    // each lane writes its own row: whole 32-byte sectors in
                    // 256-bit stores, no staging (the freed shared memory is a
                    // sixth pipeline stage)
                    if (valid) {
                        // G and U of the 32 columns side by side in one 128-byte
                        // line of the interleaved buffer (row pitch ld_out2)
                        const int64_t ro = static_cast<int64_t>(m) * e.ld_out2 + 2 * n;
                        const int cnt = PN - n < 32 ? PN - n : 32;
                        store_row32(e.out2, ro, 0, cnt, 0, v);
                        store_row32(e.out2, ro + 32, 0, cnt, 0, u);
                    }
#pragma unroll
                    for (int i = 0; i < 32; i += 2) {   // SiLU(g) * u on the bf16-rounded G and U
                        const float2 g = make_float2(round_bf16(v[i]), round_bf16(v[i + 1]));
                        const float2 uu = make_float2(round_bf16(u[i]), round_bf16(u[i + 1]));
                        const float2 a = mul2(mul2(g, sigmoid2(g)), uu);
                        v[i] = a.x;
                        v[i + 1] = a.y;
                    }
                    if (valid) store_row32(e.out, static_cast<int64_t>(m) * e.ld_out, n, PN, 0, v);
                }
            } else if constexpr (EPI == EPI_SWIGLU_BWD) {
                float g[32], u[32];
#pragma unroll 1
                for (int j = 0; j < CPW; ++j) {
                    const int c = c0 + j;
                    const int n = n0 + c * 32;
                    if (n >= PN) break;
                    // this row's [G 32 | U 32] line (loaded during the previous chunk)
#pragma unroll
                    for (int k = 0; k < 4; ++k) {
                        const uint32_t a4[4] = {gu[k].x, gu[k].y, gu[k].z, gu[k].w};
                        const uint32_t b4[4] = {gu[k + 4].x, gu[k + 4].y, gu[k + 4].z, gu[k + 4].w};
#pragma unroll
                        for (int q2 = 0; q2 < 4; ++q2) {
                            g[8 * k + 2 * q2] = bf16_lo(a4[q2]);
                            g[8 * k + 2 * q2 + 1] = bf16_hi(a4[q2]);
                            u[8 * k + 2 * q2] = bf16_lo(b4[q2]);
                            u[8 * k + 2 * q2 + 1] = bf16_hi(b4[q2]);
                        }
                    }
                    if (valid && j + 1 < CPW && n + 32 < PN)
                        load_line128(static_cast<const uint16_t*>(pa) + ra + 2 * (n + 32), gu);
                    tmem_load32(tbase + c * 32, v);
                    if (valid) {
                        float du[32];
#pragma unroll
                        for (int i = 0; i < 32; i += 2) {
                            // dU = dA SiLU(g), dG = dA u SiLU'(g), SiLU'(g) = s (1 + g (1 - s))
                            const float2 gg = make_float2(g[i], g[i + 1]);
                            const float2 sg = sigmoid2(gg);
                            const float2 vs = mul2(make_float2(v[i], v[i + 1]), sg);
                            const float2 d_u = mul2(vs, gg);
                            const float2 k = fma2(gg, add2(make_float2(1.0f, 1.0f), make_float2(-sg.x, -sg.y)),
                                                  make_float2(1.0f, 1.0f));
                            const float2 d_g = mul2(mul2(vs, make_float2(u[i], u[i + 1])), k);
                            du[i] = d_u.x;
                            du[i + 1] = d_u.y;
                            v[i] = d_g.x;
                            v[i + 1] = d_g.y;
                        }
                        store_row32(e.out, static_cast<int64_t>(m) * e.ld_out, n, PN, e.out_f32, v);
                        store_row32(e.out2, static_cast<int64_t>(m) * e.ld_out2, n, PN, e.out2_f32, du);
                    }
                }
            }
            tc_fence_before();
            if constexpr (CG == 2) {
                // one arrival per CTA on the even CTA's barrier once all 8 epilogue warps are done
                named_bar_sync(1, 256);
                if (warp == 2 && lane == 0) mbar_arrive_cluster(mapa_shared(smem_u32(&tempty[acc]), 0));
            } else {
                mbar_arrive(&tempty[acc]);
            }
        }
    }

    __syncthreads();
    if constexpr (CG == 2) cluster_sync();   // no remote arrival, load or UMMA is still in flight
    if (warp == 1) {
        __syncwarp();
        tc_fence_after();
        if constexpr (CG == 2)
            tmem_dealloc_pair(tmem_base, C::TMEM_COLS);
        else
            tmem_dealloc(tmem_base, C::TMEM_COLS);
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
                     uint32_t box_inner, uint32_t box_outer,
                     CUtensorMapSwizzle swizzle = CU_TENSOR_MAP_SWIZZLE_128B) {
    auto fn = encode_fn();
    if (!fn) return false;
    if ((reinterpret_cast<uintptr_t>(ptr) & 15u) != 0) return false;
    if ((ld * 2) % 16 != 0 || inner < 1 || outer < 1 || ld < inner) return false;
    cuuint64_t dims[2] = {static_cast<cuuint64_t>(inner), static_cast<cuuint64_t>(outer)};
    cuuint64_t strides[1] = {static_cast<cuuint64_t>(ld * 2)};
    cuuint32_t box[2] = {box_inner, box_outer};
    cuuint32_t estr[2] = {1, 1};
    CUresult r = fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(ptr), dims, strides, box, estr,
                    CU_TENSOR_MAP_INTERLEAVE_NONE, swizzle, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                    CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    return r == CUDA_SUCCESS;
}

static bool map_operand(CUtensorMap* map, const Operand& o, int64_t rows, int64_t K, uint32_t rows_box) {
    if (o.mn_major) return make_map(map, o.ptr, rows, K, o.ld, 64, 64);
    return make_map(map, o.ptr, K, rows, o.ld, 64, rows_box);
}

template <int CG, bool A_MN, bool B_MN, int EPI, int BNT = BN>
static int launch_inst(const Params& p, cudaStream_t stream) {
    using C = Cfg<CG, EPI, BNT>;
    auto k = gemm_kernel<CG, A_MN, B_MN, EPI, BNT>;
    // Resident tile walkers: CTAs (CG = 1) or CTA pairs (CG = 2) that fit at
    // once, found (and the kernel's shared-memory attribute set, which is a
    // per-device setting) on the first launch on each device.
    constexpr int kMaxDev = 64;
    static std::atomic<int> units_dev[kMaxDev];
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDev) return BOM_ECUDA;
    int max_units = units_dev[dev].load(std::memory_order_relaxed);
    if (max_units == 0) {
        if (cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, C::SMEM) != cudaSuccess)
            return BOM_ECUDA;
        if constexpr (CG == 2) {
            cudaLaunchConfig_t cfg = {};
            cfg.gridDim = dim3(static_cast<unsigned>(device_sm_count() & ~1));
            cfg.blockDim = dim3(NUM_THREADS);
            cfg.dynamicSmemBytes = C::SMEM;
            cudaLaunchAttribute at;
            at.id = cudaLaunchAttributeClusterDimension;
            at.val.clusterDim.x = 2;
            at.val.clusterDim.y = 1;
            at.val.clusterDim.z = 1;
            cfg.attrs = &at;
            cfg.numAttrs = 1;
            int n = 0;
            if (cudaOccupancyMaxActiveClusters(&n, k, &cfg) != cudaSuccess || n < 1) {
                cudaGetLastError();
                n = device_sm_count() / 2;
            }
            max_units = n;
        } else {
            max_units = device_sm_count();
        }
        units_dev[dev].store(max_units, std::memory_order_relaxed);
    }
    const int work = p.tile_base[p.nprob] * p.ksplit;
    const int units = work < max_units ? work : max_units;
    if constexpr (CG == 2) {
        cudaLaunchConfig_t cfg = {};
        cfg.gridDim = dim3(static_cast<unsigned>(2 * units));
        cfg.blockDim = dim3(NUM_THREADS);
        cfg.dynamicSmemBytes = C::SMEM;
        cfg.stream = stream;
        cudaLaunchAttribute at[2];
        at[0].id = cudaLaunchAttributeClusterDimension;
        at[0].val.clusterDim.x = 2;
        at[0].val.clusterDim.y = 1;
        at[0].val.clusterDim.z = 1;
        at[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
        at[1].val.programmaticStreamSerializationAllowed = 1;
        cfg.attrs = at;
        cfg.numAttrs = 2;
        if (cudaLaunchKernelEx(&cfg, k, p) != cudaSuccess) return BOM_ECUDA;
    } else {
        launch_k(k, dim3(units), dim3(NUM_THREADS), C::SMEM, stream, p);
    }
    count_launch();
    return cudaPeekAtLastError() == cudaSuccess ? BOM_OK : BOM_ECUDA;
}

// Split-K reduction: sums the fp32 partial slices in a fixed order and applies
// the GEMM's linear epilogue.
__global__ void __launch_bounds__(256) splitk_reduce_kernel(const float* __restrict__ ws, int S, int M, int N,
                                                            const EpiParams e) {
    pdl_enter();
    if (e.sc != nullptr && e.sc->status != 0) return;
    const int64_t total = static_cast<int64_t>(M) * N;
    const int64_t stride = static_cast<int64_t>(gridDim.x) * blockDim.x;
    for (int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; i < total; i += stride) {
        float acc = 0.0f;
        for (int s = 0; s < S; ++s) acc += ws[s * total + i];
        const int m = static_cast<int>(i / N), n = static_cast<int>(i - static_cast<int64_t>(m) * N);
        const EpiRow r = epi_row(e, m, M);
        const int64_t idx = static_cast<int64_t>(m) * e.ld_out + n;
        float v = epi_linear1(e, r, m, n, acc);
        if (e.upd_theta) v = fused_update1(e, idx, v);
        st_elem(e.out, idx, e.out_f32, v);
    }
}

// Raster of a GEMM's tiles.  The persistent walkers take tiles in order, so
// the tiles in flight at once are a window of consecutive tile indices; the
// operand panels they read are shared in L2 only while all their readers run
// together.  A GEMM at most 8 tiles wide (the weight gradients, input
// cotangents and down projection of the step, all with long K: 8 MB panels
// and more) walks whole rows of tiles, so every A panel's readers are
// consecutive and run in the same wave; wider GEMMs keep groups of 8 m-tiles,
// m fastest, so a window of tiles reads about as many A panels as B panels.
static int raster_group(int tiles_m, int tiles_n) { return tiles_n <= 8 ? 1 : GROUP_M; }

// Number of K ranges for a GEMM with `tiles` output tiles on `units` resident
// tile walkers.  GEMMs that keep the GPU at least 75% busy are not split (the
// fp32 partials cost more than milder quantisation does).  Otherwise the
// split minimises an estimate of the time in k-block steps: waves x (k-blocks
// per range + 2 for storing a tile), plus for a split the reduction (about 14
// steps of launch and fixed cost, and the partials' round trip through memory
// at about 5e-6 steps per fp32 element); among 2..8 ranges of at least 8
// k-blocks whose partials fit the scratch, the cheapest that saves 10% over
// no split.
static int choose_split(int tiles, int units, int kb_total, int64_t mn, int64_t ws_elems) {
    auto waves = [&](int s) { return (static_cast<int64_t>(tiles) * s + units - 1) / units; };
    if (static_cast<double>(tiles) / (static_cast<double>(waves(1)) * units) >= 0.75) return 1;
    auto cost = [&](int s) {
        const double per = std::ceil(static_cast<double>(kb_total) / s) + 2.0;
        double c = static_cast<double>(waves(s)) * per;
        if (s > 1) c += 14.0 + 5e-6 * static_cast<double>(s) * static_cast<double>(mn);
        return c;
    };
    const double c1 = cost(1);
    int best = 1;
    double best_cost = c1;
    for (int s = 2; s <= 8; ++s) {
        if (kb_total / s < 8 || static_cast<int64_t>(s) * mn > ws_elems) break;
        const double c = cost(s);
        if (c < 0.9 * c1 && c < best_cost) {
            best = s;
            best_cost = c;
        }
    }
    return best;
}

// Narrow single-CTA tiles: the linear epilogue with A K-major (the forward
// layers and the input cotangents of the small configurations), or with both
// operands MN-major (their weight gradients, K = the batch rows), and the
// fused update of those weight gradients.
static int dispatch_narrow(const Params& p, bool a_mn, bool b_mn, cudaStream_t stream, int epi_kind = EPI_LINEAR) {
    if (epi_kind == EPI_UPDATE)
        return a_mn && b_mn ? launch_inst<1, true, true, EPI_UPDATE, kBnSmall>(p, stream) : BOM_ENOTSUP;
    if (epi_kind != EPI_LINEAR) return BOM_ENOTSUP;
    if (a_mn) return b_mn ? launch_inst<1, true, true, EPI_LINEAR, kBnSmall>(p, stream) : BOM_ENOTSUP;
    return b_mn ? launch_inst<1, false, true, EPI_LINEAR, kBnSmall>(p, stream)
                : launch_inst<1, false, false, EPI_LINEAR, kBnSmall>(p, stream);
}

template <int CG>
static int dispatch(const Params& p, int epi_kind, bool a_mn, bool b_mn, bool dual_b, cudaStream_t stream) {
    switch (epi_kind) {
        case EPI_LINEAR:
            if (!a_mn && !b_mn) return launch_inst<CG, false, false, EPI_LINEAR>(p, stream);
            if (!a_mn && b_mn) return launch_inst<CG, false, true, EPI_LINEAR>(p, stream);
            if (a_mn && b_mn) return launch_inst<CG, true, true, EPI_LINEAR>(p, stream);
            return launch_inst<CG, true, false, EPI_LINEAR>(p, stream);
        case EPI_LOGITS:
            if (a_mn || b_mn) return BOM_ENOTSUP;
            return launch_inst<CG, false, false, EPI_LOGITS>(p, stream);
        case EPI_SWIGLU_FWD:
            if (a_mn || b_mn || !dual_b) return BOM_ENOTSUP;
            return launch_inst<CG, false, false, EPI_SWIGLU_FWD>(p, stream);
        case EPI_SWIGLU_BWD:
            if (a_mn || !b_mn) return BOM_ENOTSUP;
            return launch_inst<CG, false, true, EPI_SWIGLU_BWD>(p, stream);
        case EPI_UPDATE:   // weight gradients: dy^T x, both operands MN-major
            if (!a_mn || !b_mn) return BOM_ENOTSUP;
            return launch_inst<CG, true, true, EPI_UPDATE>(p, stream);
        default:
            return BOM_EINVAL;
    }
}

}  // namespace tc

// Cached per device ordinal (atomics: concurrent first calls from several
// host threads store the same value).
int device_sm_count() {
    constexpr int kMaxDev = 64;
    static std::atomic<int> cached[kMaxDev];
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) {
        cudaGetLastError();
        dev = 0;
    }
    int n = (dev >= 0 && dev < kMaxDev) ? cached[dev].load(std::memory_order_relaxed) : 0;
    if (n == 0) {
        if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) {
            cudaGetLastError();
            n = 0;
        }
        if (n <= 0) n = 1;
        if (dev >= 0 && dev < kMaxDev) cached[dev].store(n, std::memory_order_relaxed);
    }
    return n;
}

int64_t tc_logit_tiles(int64_t N) { return 2 * ((N + tc::BN - 1) / tc::BN); }  // one pair per column half

int launch_gemm_tc(const GemmDesc& g, cudaStream_t stream) {
    using namespace tc;
    if (g.M <= 0 || g.N <= 0) return BOM_OK;
    if (g.M > INT32_MAX / 2 || g.N > INT32_MAX / 2) return BOM_ENOTSUP;
    if (g.epi.in_f32) return BOM_ENOTSUP;   // epilogue operands are bf16 on this engine
    const bool a_mn = g.A[0].mn_major, b_mn = g.B[0].mn_major;
    // CTA pairs (256-row tiles) whenever there is more than one 128-row tile,
    // unless the 256-column tiles would leave three quarters of the SMs idle:
    // then single CTAs with 128 x 64 tiles (linear epilogue, A K-major).
    const int64_t wide_ctas = ((g.M + BM - 1) / BM) * ((g.N + BN - 1) / BN);
    const bool narrow = g.epi_kind == EPI_LINEAR && !g.dual_b && !a_mn && 4 * wide_ctas <= device_sm_count();
    const int cg = (g.M > BM && !narrow) ? 2 : 1;
    Params p;
    memset(&p, 0, sizeof(p));
    // B rows one CTA loads per stage
    const uint32_t b_rows = narrow ? kBnSmall : (cg == 2 || g.dual_b) ? 128 : 256;
    for (int s = 0; s < g.nseg; ++s) {
        if (g.A[s].mn_major != a_mn || g.B[s].mn_major != b_mn) return BOM_ENOTSUP;
        p.kb[s] = static_cast<int>((g.K[s] + BK - 1) / BK);
        if (g.K[s] <= 0) continue;
        if (!map_operand(&p.mapA[s], g.A[s], g.M, g.K[s], BM)) return BOM_ENOTSUP;
        if (g.dual_b) {
            if (b_mn || g.nseg != 1) return BOM_ENOTSUP;
            if (!map_operand(&p.mapB[0], g.B[0], g.N, g.K[0], 128)) return BOM_ENOTSUP;
            if (!map_operand(&p.mapB[1], g.B[1], g.N, g.K[0], 128)) return BOM_ENOTSUP;
        } else if (!map_operand(&p.mapB[s], g.B[s], g.N, g.K[s], b_rows)) {
            return BOM_ENOTSUP;
        }
    }
    p.M = static_cast<int>(g.M);
    p.N = static_cast<int>(g.N);
    p.nseg = g.nseg;
    p.dual_b = g.dual_b ? 1 : 0;
    p.bn_out = narrow ? kBnSmall : g.dual_b ? 128 : BN;
    p.tiles_m = static_cast<int>((g.M + BM * cg - 1) / (BM * cg));
    p.tiles_n = static_cast<int>((g.N + p.bn_out - 1) / p.bn_out);
    p.group_m = raster_group(p.tiles_m, p.tiles_n);
    p.epi = g.epi;
    const int kb_total = p.kb[0] + (p.nseg > 1 ? p.kb[1] : 0);
    const int tiles = p.tiles_m * p.tiles_n;
    p.nprob = 1;
    p.tile_base[0] = 0;
    p.tile_base[1] = tiles;
    const int units = cg == 2 ? device_sm_count() / 2 : device_sm_count();
    int S = 1;
    // (column sums are formed in the tile epilogue: no split)
    if ((g.epi_kind == EPI_LINEAR || g.epi_kind == EPI_UPDATE) && g.splitk_ws != nullptr && g.epi.colsum == nullptr)
        S = choose_split(tiles, units, kb_total, static_cast<int64_t>(g.M) * g.N, g.splitk_ws_elems);
    p.ksplit = S;
    p.kb_split = S > 1 ? (kb_total + S - 1) / S : kb_total;
    if (S > 1) {
        // raw fp32 partial tiles into the scratch; the real epilogue runs in the reduction
        p.ksplit = (kb_total + p.kb_split - 1) / p.kb_split;
        EpiParams raw = {};
        raw.alpha_const = 1.0f;
        raw.beta_const = 0.0f;
        raw.out = g.splitk_ws;
        raw.ld_out = g.N;
        raw.out_f32 = 1;
        raw.sc = g.epi.sc;
        p.epi = raw;
        p.split_bytes = static_cast<int64_t>(g.M) * g.N * 4;
    }
    // split-K partial tiles are raw (linear epilogue); the update, if any,
    // runs in the reduction
    const int kind = S > 1 ? EPI_LINEAR : g.epi_kind;
    const int rc = narrow    ? dispatch_narrow(p, a_mn, b_mn, stream)
                   : cg == 2 ? dispatch<2>(p, kind, a_mn, b_mn, g.dual_b, stream)
                             : dispatch<1>(p, kind, a_mn, b_mn, g.dual_b, stream);
    if (rc != BOM_OK || S == 1) return rc;
    const int64_t total = static_cast<int64_t>(g.M) * g.N;
    int64_t blocks = (total + 255) / 256;
    if (blocks > 8 * device_sm_count()) blocks = 8 * device_sm_count();
    launch_k(splitk_reduce_kernel, dim3(static_cast<unsigned>(blocks)), dim3(256), 0, stream, g.splitk_ws, p.ksplit, p.M, p.N, g.epi);
    count_launch();
    return cudaPeekAtLastError() == cudaSuccess ? BOM_OK : BOM_ECUDA;
}

}  // namespace bom

namespace bom {

// One persistent launch over up to kMaxGroup GEMMs that share the operand
// layout, the epilogue kind and K (the weight gradients of a SwiGLU sublayer,
// with the head's): their tiles form one work list, so the last wave is
// shared instead of each GEMM ending on its own partial wave.  Falls back to
// separate launches when the GEMMs do not fit one launch.
int launch_gemm_tc_group(const GemmDesc* gs, int n, cudaStream_t stream) {
    using namespace tc;
    bool ok = n >= 1 && n <= kMaxGroup;
    for (int i = 0; ok && i < n; ++i) {
        const GemmDesc& g = gs[i];
        ok = g.nseg == 1 && !g.dual_b && !g.epi.in_f32 && g.M > BM && g.N > 0 && g.K[0] == gs[0].K[0] &&
             g.epi_kind == gs[0].epi_kind && g.A[0].mn_major == gs[0].A[0].mn_major &&
             g.B[0].mn_major == gs[0].B[0].mn_major && g.M <= INT32_MAX / 2 && g.N <= INT32_MAX / 2;
    }
    if (!ok) {
        for (int i = 0; i < n; ++i) {
            const int rc = launch_gemm_tc(gs[i], stream);
            if (rc != BOM_OK) return rc;
        }
        return BOM_OK;
    }
    Params p;
    memset(&p, 0, sizeof(p));
    const GemmDesc& g0 = gs[0];
    p.kb[0] = static_cast<int>((g0.K[0] + BK - 1) / BK);
    // Weight gradients over a short K (at most 16 k-blocks: small batches)
    // with a linear epilogue (u to memory) or the fused update spend most of a
    // 256 x 256 tile in its epilogue, and their few hundred tiles end on a
    // partial wave of CTA pairs: single CTAs with 128 x 64 tiles instead.
    const bool narrow = (g0.epi_kind == EPI_LINEAR || g0.epi_kind == EPI_UPDATE) && p.kb[0] <= 16 &&
                        g0.A[0].mn_major && g0.B[0].mn_major;
    const int tile_m = narrow ? BM : 2 * BM, tile_n = narrow ? kBnSmall : BN;
    p.nseg = 1;
    p.bn_out = tile_n;
    p.ksplit = 1;
    p.kb_split = p.kb[0];
    p.nprob = n;
    int tiles = 0;
    for (int i = 0; i < n; ++i) {
        const GemmDesc& g = gs[i];
        CUtensorMap* ma = i == 0 ? &p.mapA[0] : &p.grp[i - 1].mapA;
        CUtensorMap* mb = i == 0 ? &p.mapB[0] : &p.grp[i - 1].mapB;
        if (g.K[0] > 0 && (!map_operand(ma, g.A[0], g.M, g.K[0], BM) ||
                           !map_operand(mb, g.B[0], g.N, g.K[0], narrow ? kBnSmall : 128)))
            return BOM_ENOTSUP;
        const int tm = static_cast<int>((g.M + tile_m - 1) / tile_m);
        const int tn = static_cast<int>((g.N + tile_n - 1) / tile_n);
        if (i == 0) {
            p.M = static_cast<int>(g.M);
            p.N = static_cast<int>(g.N);
            p.tiles_m = tm;
            p.tiles_n = tn;
            p.group_m = raster_group(tm, tn);
            p.epi = g.epi;
        } else {
            Prob& q = p.grp[i - 1];
            q.M = static_cast<int>(g.M);
            q.N = static_cast<int>(g.N);
            q.tiles_m = tm;
            q.tiles_n = tn;
            q.group_m = raster_group(tm, tn);
            q.epi = g.epi;
        }
        p.tile_base[i] = tiles;
        tiles += tm * tn;
    }
    p.tile_base[n] = tiles;
    if (narrow) return dispatch_narrow(p, true, true, stream, g0.epi_kind);
    return dispatch<2>(p, g0.epi_kind, g0.A[0].mn_major, g0.B[0].mn_major, false, stream);
}

}  // namespace bom
