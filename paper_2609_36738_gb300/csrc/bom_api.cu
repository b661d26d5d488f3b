// C ABI of the BOM task-space momentum pass: handle and workspace, argument
// checks, and the orchestration of one step (Algorithm 1) as a sequence of
// stream-ordered kernels.  Nothing here synchronises except bom_get_stats.
//
// Step, for a batch of n rows (paper: Algorithm 1; Section 3.2):
//   forward   backbone GEMMs with fused bias/GELU/SwiGLU/residual epilogues,
//             logits GEMM Z = H W^T (+b) whose epilogue stores Z and per-tile
//             (max, sum exp) row statistics;
//   task      label scan (N_t), row log-sum-exp, residual pass Z -> R with
//             column partial sums, s_t, q_t = beta1 q + (1-beta1) s_t,
//             qhat_t = q_t / (1-beta1^t), c = colsum_{I_t}(H), w = W^T qhat;
//   backward  head dW = a R^T H + b qhat (x) c      (rank-1 epilogue),
//             head dH = a R W + b 1_{I_t} w^T       (broadcast-row epilogue),
//             then the backbone VJPs, with (a, b) = N_t^-1 (1-lambda, lambda)
//             for u, N_t^-1 (1, 0) for g and N_t^-1 (0, 1) for h; the
//             own-step pass (telemetry) broadcasts s_t in place of qhat.
// With the fused update registered, each weight is updated in the epilogue of
// the GEMM that forms its u (the weight gradients of a block run as one
// grouped launch after its last input cotangent), and each vector right
// after its gradient.  The step's scalars (lr, 1/(1-beta1^t), 1/(1-beta2^t))
// live in the device scalar block, written by the label scan from the host's
// values or from a registered device step counter, so a captured step
// (bom_graph_capture) replays correctly for every later t.
#include <cmath>
#include <cstdlib>
#include <cstring>
#include <new>
#include <atomic>
#include <vector>

#include <nvtx3/nvToolsExt.h>

#include "gemm.h"
#include "kernels.h"

using namespace bom;

namespace {

struct LayerWs {
    int kind = 0;
    int64_t d_in = 0, d_out = 0;
    bool bias = false;
    int64_t width_out = 0;   // width of the layer output
    void* pre = nullptr;     // LINEAR_GELU pre-activation [n, d_out]
    void* out = nullptr;     // layer output [n, width_out]
    void* G = nullptr;       // SWIGLU gate and up pre-activations, interleaved per 32
                             // columns: [G 32 | U 32] blocks, row pitch gu_ld
    int64_t gu_ld = 0;       // 2 * ffn rounded up to 64
    void* A = nullptr;       // SWIGLU SiLU(G) * U [n, ffn]
    float* rstd = nullptr;   // RMSNORM 1 / sqrt(mean x^2 + eps) per row [n]
    // a biased Linear layer of a small batch (bf16): fp32 column sums of its
    // output cotangent per 32-row block [ceil(n / 32), d_out], written by the
    // epilogue of the GEMM that produces the cotangent
    float* cspart = nullptr;
};

int64_t round_up(int64_t a, int64_t b) { return (a + b - 1) / b * b; }

// Rows up to which a step with the update registered writes u and updates
// every tensor in one streaming launch instead of in the weight-gradient
// GEMMs' epilogues (see bom_handle::uscr).
constexpr int64_t kUpdSepRows = 1024;

}  // namespace

struct bom_handle {
    bom_config cfg{};
    std::vector<bom_layer> layers;
    std::vector<LayerWs> lw;
    bool bf16 = false;
    int64_t esz = 4;
    int64_t d_model = 0;
    int64_t max_width = 0;
    int64_t max_ffn = 0;
    char* ws = nullptr;
    size_t ws_bytes = 0;
    DevScalars* sc = nullptr;
    void* Z = nullptr;
    int64_t ldz = 0;
    float* stats = nullptr;
    int64_t ntiles = 1;
    float* lse = nullptr;
    float* ce = nullptr;
    float* colpart = nullptr;
    float* s = nullptr;
    float* qhat = nullptr;
    float* cvec = nullptr;
    float* wvec = nullptr;
    float* wsvec = nullptr;  // W^T s_t (own-step pass)
    float* rnorm = nullptr;  // ||r_i|| per row (own-step telemetry)
    double* tel_part = nullptr;  // per-block partials of bom_own_step_moment
    std::vector<void*> own_out;  // own-step projection outputs (bom_set_own_step_output)
    // fused BOM-AdamW update (bom_set_fused_update)
    bool fused_upd = false;
    std::vector<float*> upd_theta, upd_v;
    std::vector<float> upd_wd;
    float upd_lr = 0.0f, upd_beta2 = 0.0f, upd_eps = 0.0f;
    // device step scalars (bom_set_step_scalars): t and lr read by the step's kernels
    int64_t* t_dev = nullptr;
    const float* lr_dev = nullptr;
    float* ubuf = nullptr;   // fp32 u of a vector tensor (bias, norm weight) before its update
    // Small batches (max_rows <= kUpdSepRows): fp32 u of every tensor, so
    // that a step with the update registered writes u from the weight-gradient
    // GEMMs and updates all tensors in one streaming launch (with a K of a few
    // hundred rows the update epilogue of those GEMMs is latency-bound).
    float* uscr = nullptr;
    std::vector<int64_t> uoff, unum;   // per tensor: offset in uscr (16-byte aligned), elements
    float* part = nullptr;
    void* dx[2] = {nullptr, nullptr};
    void* dG = nullptr;
    void* dU = nullptr;
    void* dG2 = nullptr;     // the second sublayer's dG, dU while its weight gradients wait
    void* dU2 = nullptr;
    void* dx_in = nullptr;   // caller buffer for the cotangent of X (bom_set_input_grad)
    float* splitk = nullptr; // fp32 partial tiles of split-K GEMMs
    int64_t splitk_elems = 0;
    int64_t last_n = 0;
    int64_t shard_n = 0;     // rows of the first half of a sharded step (0: none pending)
    float* sshard = nullptr; // this shard's s^shard = N_t^-1 sum_{i in I_t^shard} r_i (sharded steps)
    // vocabulary-sharded step: the whole vocabulary, this shard's first id, the
    // rows of the step in progress and how far it got (0 none, 1 after begin,
    // 2 after mid)
    int64_t vs_total = 0, vs_first = 0, vs_n = 0;
    int vs_stage = 0;
    // tracing: one event pair per launch of the current step
    struct TraceRec {
        const char* name = nullptr;
        double flops = 0, bytes = 0;
        cudaEvent_t a = nullptr, b = nullptr;
    };
    std::vector<TraceRec> trace;
    int trace_n = 0;
    bool tracing = false;
};

namespace bom {
static std::atomic<long long> g_launches{0};
void count_launch() { g_launches.fetch_add(1, std::memory_order_relaxed); }
}  // namespace bom

namespace {

bom_status check_config(const bom_config* cfg, std::vector<LayerWs>* lw_out, int64_t* d_model, int64_t* max_width,
                        int64_t* max_ffn) {
    if (!cfg) return BOM_EINVAL;
    if (cfg->max_rows < 1 || cfg->d_in < 1 || cfg->d_out < 1 || cfg->n_layers < 0) return BOM_EINVAL;
    if (cfg->n_layers > 0 && !cfg->layers) return BOM_EINVAL;
    if (cfg->compute != BOM_F32 && cfg->compute != BOM_BF16) return BOM_EINVAL;
    if (cfg->out_mode != BOM_OUT_U && cfg->out_mode != BOM_OUT_G_AND_H) return BOM_EINVAL;
    if (!(cfg->lambda >= 0.0f && cfg->lambda <= 1.0f)) return BOM_EINVAL;
    if (!(cfg->beta1 >= 0.0f && cfg->beta1 < 1.0f)) return BOM_EINVAL;
    if (cfg->max_rows > (1ll << 30) || cfg->d_out > (1ll << 30)) return BOM_ENOTSUP;
    // The residual pass and the fp32 GEMM put 64-row blocks on gridDim.y (at
    // most 65535 blocks): refused here, before any step could stop half done.
    constexpr int64_t kMaxGridRows = static_cast<int64_t>(kResidRows) * 65535;
    if (cfg->max_rows > kMaxGridRows) return BOM_ENOTSUP;
    const bool bf16 = cfg->compute == BOM_BF16;
    std::vector<LayerWs> lw;
    int64_t w = cfg->d_in, mw = cfg->d_in, mf = 0;
    for (int i = 0; i < cfg->n_layers; ++i) {
        const bom_layer& L = cfg->layers[i];
        LayerWs x;
        x.kind = L.kind;
        x.d_in = L.d_in;
        x.d_out = L.d_out;
        x.bias = L.has_bias != 0;
        if (L.d_in != w || L.d_out < 1) return BOM_EINVAL;
        if (L.kind == BOM_LAYER_SWIGLU) {
            if (L.has_bias) return BOM_EINVAL;
            if (!bf16) return BOM_ENOTSUP;
            x.width_out = L.d_in;
            mf = mf > L.d_out ? mf : L.d_out;
        } else if (L.kind == BOM_LAYER_LINEAR || L.kind == BOM_LAYER_LINEAR_GELU) {
            x.width_out = L.d_out;
        } else if (L.kind == BOM_LAYER_RMSNORM) {
            if (L.has_bias || L.d_out != L.d_in) return BOM_EINVAL;
            x.width_out = L.d_in;
        } else {
            return BOM_EINVAL;
        }
        w = x.width_out;
        mw = mw > w ? mw : w;
        mw = mw > L.d_out ? mw : L.d_out;
        lw.push_back(x);
    }
    if (bf16) {
        // TMA needs 16-byte row pitches: every width must be a multiple of 8.
        if (cfg->d_in % 8) return BOM_ENOTSUP;
        for (auto& x : lw)
            if (x.d_out % 8 || x.d_in % 8) return BOM_ENOTSUP;
    } else {
        // fp32 weight gradients run with M = the output width of the head or layer
        if (cfg->d_out > kMaxGridRows) return BOM_ENOTSUP;
        for (auto& x : lw)
            if (x.d_out > kMaxGridRows) return BOM_ENOTSUP;
    }
    *d_model = w;
    *max_width = mw;
    *max_ffn = mf;
    if (lw_out) *lw_out = lw;
    return BOM_OK;
}

struct Carver {
    size_t off = 0;
    char* base = nullptr;
    void* take(size_t bytes) {
        off = (off + 255) & ~size_t(255);
        void* p = base ? base + off : nullptr;
        off += bytes;
        return p;
    }
};

// Lays out (base == nullptr: only measures) the workspace of a handle.
size_t carve(bom_handle* h, char* base) {
    Carver c;
    c.base = base;
    const int64_t n = h->cfg.max_rows, V = h->cfg.d_out, e = h->esz;
    h->sc = static_cast<DevScalars*>(c.take(sizeof(DevScalars)));
    for (auto& L : h->lw) {
        if (L.kind == BOM_LAYER_SWIGLU) {
            // G and U of each 32 columns share one 128-byte line of a row: the
            // forward writes whole lines, the backward epilogue reads one box
            L.gu_ld = 2 * round_up(L.d_out, 32);
            L.G = c.take(n * L.gu_ld * e);
            L.A = c.take(n * L.d_out * e);
        } else if (L.kind == BOM_LAYER_LINEAR_GELU) {
            L.pre = c.take(n * L.d_out * e);
        } else if (L.kind == BOM_LAYER_RMSNORM) {
            L.rstd = static_cast<float*>(c.take(n * 4));
        }
        if (h->bf16 && L.bias && n <= kUpdSepRows && (L.kind == BOM_LAYER_LINEAR || L.kind == BOM_LAYER_LINEAR_GELU))
            L.cspart = static_cast<float*>(c.take((n + 31) / 32 * L.d_out * 4));
        L.out = c.take(n * L.width_out * e);
    }
    // logits rows start on 128-byte boundaries: each 64-byte row segment an
    // epilogue warp stores then covers whole 32-byte sectors (no partial-sector
    // merges in L2) and the residual pass reads aligned lines
    h->ldz = round_up(V, h->bf16 ? 64 : 32);
    h->Z = c.take(n * h->ldz * e);
    h->ntiles = h->bf16 ? tc_logit_tiles(V) : 1;
    h->stats = static_cast<float*>(c.take(n * h->ntiles * 8));
    h->lse = static_cast<float*>(c.take(n * 4));
    h->ce = static_cast<float*>(c.take(n * 4));
    h->colpart = static_cast<float*>(c.take(resid_blocks(n) * V * 4));
    h->s = static_cast<float*>(c.take(V * 4));
    h->qhat = static_cast<float*>(c.take(V * 4));
    h->sshard = static_cast<float*>(c.take(V * 4));
    h->cvec = static_cast<float*>(c.take(h->d_model * 4));
    h->wvec = static_cast<float*>(c.take(h->d_model * 4));
    h->wsvec = static_cast<float*>(c.take(h->d_model * 4));
    h->rnorm = static_cast<float*>(c.take(n * 4));
    h->tel_part = static_cast<double*>(c.take(4 * kOwnStepMaxBlocks * sizeof(double)));
    h->ubuf = static_cast<float*>(c.take((V > h->max_width ? V : h->max_width) * 4));
    if (n <= kUpdSepRows) {
        const int np = bom_param_count(&h->cfg);
        h->uoff.assign(np, 0);
        h->unum.assign(np, 0);
        int64_t tot = 0;
        for (int k = 0; k < np; ++k) {
            int64_t r = 0, cc = 0;
            bom_param_shape(&h->cfg, k, &r, &cc);
            h->unum[k] = r * (cc > 0 ? cc : 1);
            h->uoff[k] = tot;
            tot += round_up(h->unum[k], 4);
        }
        h->uscr = np <= kMultiUpdMax ? static_cast<float*>(c.take(tot * 4)) : nullptr;
        if (np > kMultiUpdMax) h->uoff.clear();
    }
    const int64_t rb = row_blocks(n) > row_blocks(V) ? row_blocks(n) : row_blocks(V);
    h->part = static_cast<float*>(c.take(rb * h->max_width * 4));
    h->dx[0] = c.take(n * h->max_width * e);
    h->dx[1] = c.take(n * h->max_width * e);
    if (h->max_ffn > 0) {
        h->dG = c.take(n * h->max_ffn * e);
        h->dU = c.take(n * h->max_ffn * e);
    }
    // Two SwiGLU sublayers first: the second one's weight gradients wait for
    // the first one's launch, so its dG and dU need buffers of their own.
    if (h->bf16 && h->lw.size() >= 2 && h->lw[0].kind == BOM_LAYER_SWIGLU && h->lw[1].kind == BOM_LAYER_SWIGLU) {
        h->dG2 = c.take(n * h->lw[1].d_out * e);
        h->dU2 = c.take(n * h->lw[1].d_out * e);
    }
    if (h->bf16) {
        const int64_t rows = n > V ? n : V;
        const int64_t cols = h->max_width > h->max_ffn ? h->max_width : h->max_ffn;
        const int64_t cap = int64_t(32) << 20;   // 128 MB of fp32 partials at most
        h->splitk_elems = 8 * rows * cols < cap ? 8 * rows * cols : cap;
        h->splitk = static_cast<float*>(c.take(h->splitk_elems * 4));
    }
    return c.off + 256;
}

Operand kmaj(const void* p, int64_t ld) { return Operand{p, ld, false}; }
Operand mnmaj(const void* p, int64_t ld) { return Operand{p, ld, true}; }

// Runs `launch` between an event pair when the handle traces.
template <class F>
int traced(bom_handle* h, cudaStream_t s, const char* name, double flops, double bytes, F&& launch) {
    if (!h->tracing) return launch();
    if (h->trace_n == static_cast<int>(h->trace.size())) {
        bom_handle::TraceRec r;
        if (cudaEventCreate(&r.a) != cudaSuccess || cudaEventCreate(&r.b) != cudaSuccess) return BOM_ECUDA;
        h->trace.push_back(r);
    }
    bom_handle::TraceRec& r = h->trace[h->trace_n++];
    r.name = name;
    r.flops = flops;
    r.bytes = bytes;
    nvtxRangePushA(name);   // the launch shows up under its kernel class in a profiler timeline
    cudaEventRecord(r.a, s);
    const int rc = launch();
    cudaEventRecord(r.b, s);
    nvtxRangePop();
    return rc;
}

// An NVTX range over a whole entry point (closed on every return path).
struct NvtxRange {
    explicit NvtxRange(const char* name) { nvtxRangePushA(name); }
    ~NvtxRange() { nvtxRangePop(); }
    NvtxRange(const NvtxRange&) = delete;
    NvtxRange& operator=(const NvtxRange&) = delete;
};

const char* gemm_name(const GemmDesc& g, bool bf16) {
    if (!bf16) return "gemm_simt";
    switch (g.epi_kind) {
        case EPI_LOGITS: return "gemm_tc.logits";
        case EPI_UPDATE: return "gemm_tc.update.mm";
        case EPI_SWIGLU_FWD: return "gemm_tc.swiglu_fwd";
        case EPI_SWIGLU_BWD: return "gemm_tc.swiglu_bwd";
        default: break;
    }
    const bool a = g.A[0].mn_major, b = g.B[0].mn_major;
    return a ? (b ? "gemm_tc.linear.mm" : "gemm_tc.linear.mk") : (b ? "gemm_tc.linear.km" : "gemm_tc.linear.kk");
}

int run_gemm(bom_handle* h, GemmDesc& g, cudaStream_t s) {
    g.epi.sc = h->sc;
    g.epi.in_f32 = h->bf16 ? 0 : 1;
    if (h->bf16 && (g.epi_kind == EPI_LINEAR || g.epi_kind == EPI_UPDATE)) {
        g.splitk_ws = h->splitk;
        g.splitk_ws_elems = h->splitk_elems;
    }
    double k = 0;
    for (int i = 0; i < g.nseg; ++i) k += static_cast<double>(g.K[i]);
    const double n_mma = g.dual_b ? 2.0 * g.N : static_cast<double>(g.N);
    const double flops = 2.0 * static_cast<double>(g.M) * n_mma * k;
    // output bytes per element: u, or with the fused update theta and v read
    // and written plus the compute copy
    const double out_b = g.epi.upd_theta ? 16.0 + h->esz : (g.epi.out_f32 ? 4.0 : h->esz);
    const double bytes = h->esz * (static_cast<double>(g.M) * k + n_mma * k) + out_b * static_cast<double>(g.M) * g.N;
    return traced(h, s, gemm_name(g, h->bf16), flops, bytes,
                  [&] { return h->bf16 ? launch_gemm_tc(g, s) : launch_gemm_simt(g, s); });
}

// Several GEMMs that share layout, epilogue kind and K as one launch (the
// tcgen05 path groups them into one work list; the SIMT path runs them in turn).
int run_gemm_group(bom_handle* h, GemmDesc* gs, int n, cudaStream_t s) {
    double flops = 0, bytes = 0;
    for (int i = 0; i < n; ++i) {
        GemmDesc& g = gs[i];
        g.epi.sc = h->sc;
        g.epi.in_f32 = h->bf16 ? 0 : 1;
        const double k = static_cast<double>(g.K[0]);
        flops += 2.0 * static_cast<double>(g.M) * g.N * k;
        const double out_b = g.epi.upd_theta ? 16.0 + h->esz : (g.epi.out_f32 ? 4.0 : h->esz);
        bytes += h->esz * (static_cast<double>(g.M) * k + static_cast<double>(g.N) * k) +
                 out_b * static_cast<double>(g.M) * g.N;
    }
    return traced(h, s, gemm_name(gs[0], h->bf16), flops, bytes, [&] {
        if (h->bf16) return launch_gemm_tc_group(gs, n, s);
        if (n <= 4) return launch_gemm_simt_group(gs, n, s);
        for (int i = 0; i < n; ++i) {
            const int rc = launch_gemm_simt(gs[i], s);
            if (rc != BOM_OK) return rc;
        }
        return static_cast<int>(BOM_OK);
    });
}

#define BOM_TRACED(name, flops, bytes, stmt) \
    traced(h, s, name, (flops), (bytes), [&] { stmt; return static_cast<int>(BOM_OK); })

GemmDesc gemm1(int64_t M, int64_t N, int64_t K, Operand A, Operand B) {
    GemmDesc g;
    g.M = M;
    g.N = N;
    g.K[0] = K;
    g.A[0] = A;
    g.B[0] = B;
    g.nseg = 1;
    g.epi.alpha_const = 1.0f;
    g.epi.beta_const = 1.0f;
    return g;
}

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

}  // namespace

extern "C" {

int32_t bom_param_count(const bom_config* cfg) {
    if (!cfg || cfg->n_layers < 0 || (cfg->n_layers > 0 && !cfg->layers)) return -1;
    int32_t k = 0;
    for (int i = 0; i < cfg->n_layers; ++i) {
        const bom_layer& L = cfg->layers[i];
        k += L.kind == BOM_LAYER_SWIGLU ? 3 : (L.kind == BOM_LAYER_RMSNORM ? 1 : (L.has_bias ? 2 : 1));
    }
    return k + (cfg->head_bias ? 2 : 1);
}

bom_status bom_param_shape(const bom_config* cfg, int32_t index, int64_t* rows, int64_t* cols) {
    if (!cfg || !rows || !cols || index < 0) return BOM_EINVAL;
    int32_t k = 0;
    int64_t w = cfg->d_in;
    for (int i = 0; i < cfg->n_layers; ++i) {
        const bom_layer& L = cfg->layers[i];
        if (L.kind == BOM_LAYER_SWIGLU) {
            const int64_t r[3] = {L.d_out, L.d_out, L.d_in}, c[3] = {L.d_in, L.d_in, L.d_out};
            for (int j = 0; j < 3; ++j, ++k)
                if (k == index) { *rows = r[j]; *cols = c[j]; return BOM_OK; }
        } else if (L.kind == BOM_LAYER_RMSNORM) {
            if (k++ == index) { *rows = L.d_in; *cols = 0; return BOM_OK; }
        } else {
            if (k++ == index) { *rows = L.d_out; *cols = L.d_in; return BOM_OK; }
            if (L.has_bias && k++ == index) { *rows = L.d_out; *cols = 0; return BOM_OK; }
            w = L.d_out;
        }
    }
    if (k++ == index) { *rows = cfg->d_out; *cols = w; return BOM_OK; }
    if (cfg->head_bias && k++ == index) { *rows = cfg->d_out; *cols = 0; return BOM_OK; }
    return BOM_EINVAL;
}

int64_t bom_workspace_bytes(const bom_config* cfg) {
    bom_handle h;
    int64_t dm, mw, mf;
    if (check_config(cfg, &h.lw, &dm, &mw, &mf) != BOM_OK) return -1;
    h.cfg = *cfg;
    h.bf16 = cfg->compute == BOM_BF16;
    h.esz = h.bf16 ? 2 : 4;
    h.d_model = dm;
    h.max_width = mw;
    h.max_ffn = mf;
    return static_cast<int64_t>(carve(&h, nullptr));
}

bom_status bom_init(bom_handle** out, const bom_config* cfg) {
    if (!out) return BOM_EINVAL;
    *out = nullptr;
    bom_handle* h = new (std::nothrow) bom_handle();
    if (!h) return BOM_ENOMEM;
    int64_t dm, mw, mf;
    bom_status st = check_config(cfg, &h->lw, &dm, &mw, &mf);
    if (st != BOM_OK) {
        delete h;
        return st;
    }
    h->cfg = *cfg;
    h->layers.assign(cfg->layers, cfg->layers + cfg->n_layers);
    h->cfg.layers = h->layers.data();
    h->bf16 = cfg->compute == BOM_BF16;
    h->esz = h->bf16 ? 2 : 4;
    h->d_model = dm;
    h->max_width = mw;
    h->max_ffn = mf;
    const size_t bytes = carve(h, nullptr);
    void* p = nullptr;
    if (cudaMalloc(&p, bytes) != cudaSuccess) {
        cudaGetLastError();
        delete h;
        return BOM_ENOMEM;
    }
    h->ws = static_cast<char*>(p);
    h->ws_bytes = bytes;
    carve(h, h->ws + ((256 - (reinterpret_cast<uintptr_t>(h->ws) & 255)) & 255));
    // Zero everything once: the padding columns of Z and the scalar block start defined.
    if (cudaMemset(h->ws, 0, bytes) != cudaSuccess) {
        cudaFree(p);
        delete h;
        return BOM_ECUDA;
    }
    *out = h;
    return BOM_OK;
}

void bom_destroy(bom_handle* h) {
    if (!h) return;
    if (h->ws) cudaFree(h->ws);
    for (auto& r : h->trace) {
        cudaEventDestroy(r.a);
        cudaEventDestroy(r.b);
    }
    delete h;
}

}  // extern "C"

namespace {

// The uses of one step body: a whole step, the two halves of a row-sharded
// step around the caller's sum of the exchange vector, and the three parts of
// a vocabulary-sharded step around the caller's two exchanges (the row
// log-sum-exp parts, then the head's input cotangent).
enum StepPart { kStepFull = 0, kShardBegin = 1, kShardEnd = 2, kVBegin = 3, kVMid = 4, kVEnd = 5 };
// Most shards whose row log-sum-exp parts one middle part combines.
constexpr int32_t kMaxVocabShards = 4096;

// Caller buffers of a vocabulary-sharded step (see bom_step_vshard_*).
struct VShardIo {
    float* lse_part = nullptr;        // begin: this shard's part of each row's log-sum-exp [n]
    const float* lse_parts = nullptr; // mid: every shard's part [nsh, n], in shard order
    int32_t nsh = 0;
    float* dh_part = nullptr;         // mid: this shard's part of the head's input cotangent [n, d]
    const float* dh_sum = nullptr;    // end: the shards' parts summed [n, d]
};

bom_status check_step_args(bom_handle* h, const void* x, const int32_t* labels, int64_t n, void* const* params,
                           const float* q, int64_t t, void* const* grads, void* const* h_out, int part) {
    const bool fused = h != nullptr && h->fused_upd;
    if (!h || !x || !labels || !params) return BOM_EINVAL;
    if (n < 1 || n > h->cfg.max_rows) return BOM_EINVAL;
    // a sharded step's update follows the caller's gradient sum, and the
    // own-step telemetry needs every row's residual norm
    if (part != kStepFull && (fused || !h->own_out.empty())) return BOM_EINVAL;
    // a vocabulary-sharded step has one cotangent pass (one exchange of it)
    if (part >= kVBegin && h->cfg.out_mode != BOM_OUT_U) return BOM_EINVAL;
    const int np = bom_param_count(&h->cfg);
    if (part == kShardBegin || part == kVBegin || part == kVEnd) {
        if (part == kVEnd && !grads) return BOM_EINVAL;
        for (int i = 0; i < np; ++i) {
            if (!params[i] || (part == kVEnd && !grads[i])) return BOM_EINVAL;
            if (!aligned16(params[i]) || (part == kVEnd && !aligned16(grads[i]))) return BOM_ENOTSUP;
        }
        return aligned16(x) ? BOM_OK : BOM_ENOTSUP;
    }
    if (!q || (!grads && !fused)) return BOM_EINVAL;
    if (t < 1 && h->t_dev == nullptr) return BOM_EINVAL;
    const bool gh = h->cfg.out_mode == BOM_OUT_G_AND_H;
    if (gh != (h_out != nullptr)) return BOM_EINVAL;
    // the fused update consumes u: one u pass and nothing else that needs it
    if (fused && (gh || !h->own_out.empty())) return BOM_EINVAL;
    for (int i = 0; i < np; ++i) {
        if (!params[i] || (!fused && !grads[i]) || (gh && !h_out[i])) return BOM_EINVAL;
        if (!aligned16(params[i]) || (!fused && !aligned16(grads[i])) || (gh && !aligned16(h_out[i])))
            return BOM_ENOTSUP;
    }
    if (!aligned16(x) || !aligned16(q)) return BOM_ENOTSUP;
    return BOM_OK;
}

// One step (part = kStepFull), or one half of a row-sharded step: kShardBegin
// runs the forward and the residual pass and writes this shard's exchange
// vector to xch_out; kShardEnd reads the summed vector xch_in and runs the
// rest (s_t, q_t, qhat_t, the backward of this shard's rows).  Arguments are
// checked by the caller.
bom_status step_impl(bom_handle* h, const void* x, const int32_t* labels, int64_t n, void* const* params, float* q,
                     int64_t t, void* const* grads, void* const* h_out, void* stream, int part, double* xch_out,
                     const double* xch_in, const VShardIo* vio = nullptr) {
    const bool fused = h->fused_upd;
    const bool gh = h->cfg.out_mode == BOM_OUT_G_AND_H;
    const bool shard = part == kShardBegin || part == kShardEnd;   // row-sharded
    const bool vshard = part >= kVBegin;                             // vocabulary-sharded
    // the parts that begin a step (clear the status word, restart the trace)
    const bool first_part = part == kStepFull || part == kShardBegin || part == kVBegin;
    // a small batch with the update registered: u of every tensor to the
    // scratch, then one update launch for all of them at the end of the step
    const bool upd_sep = fused && h->uscr != nullptr && n <= kUpdSepRows;
    // where the fp32 u of vector tensor k goes when the update is registered
    auto uvec = [&](int k) -> float* { return upd_sep ? h->uscr + h->uoff[k] : h->ubuf; };
    // With at most two backbone layers their output cotangents stay in the two
    // ping-pong buffers until the step ends, so for a batch of at most 128 rows
    // a Linear layer's bias gradient (their column sum) is formed by the final
    // update itself, in the order of the column reduction over one range.
    const bool fold_bias = upd_sep && h->lw.size() <= 2 && n <= kRowBlock;
    // Otherwise (bf16) the GEMM that writes a biased Linear layer's output
    // cotangent also writes its column sums per 32-row block, and the final
    // update adds those up: no column-reduction launches.
    const bool cs_fused = upd_sep && h->bf16 && !fold_bias;
    std::vector<const void*> usrc;
    std::vector<int64_t> urows;
    std::vector<int> usf32;
    if (fold_bias || cs_fused) {
        const int npar = bom_param_count(&h->cfg);
        usrc.assign(npar, nullptr);
        urows.assign(npar, n);
        usf32.assign(npar, h->bf16 ? 0 : 1);
    }
    std::vector<char> cs_ready(h->lw.size(), 0);   // per layer: its cotangent's column sums are being written
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    const bom_config& cfg = h->cfg;
    const int64_t V = cfg.d_out, dm = h->d_model;
    const int cf32 = h->bf16 ? 0 : 1;
    h->last_n = n;
    // a traced sharded step records all its parts
    if (first_part) h->trace_n = 0;
    // the second half of a sharded step needs the first half's rows in the workspace
    h->shard_n = part == kShardBegin ? n : 0;
    if (!vshard) h->vs_stage = 0;
    int rc = BOM_OK;
#define BOM_TRY(expr)                                     \
    do {                                                  \
        rc = (expr);                                      \
        if (rc != BOM_OK) return static_cast<bom_status>(rc); \
    } while (0)

    // step scalars: from the host t and lr, or from the device step counter
    // (a shard's first half has no t: its scalars are set by the second)
    StepScalarsIn st{};
    st.lr = fused ? h->upd_lr : 0.0f;
    const bool no_t = part == kShardBegin || part == kVBegin;   // first halves take no t
    st.inv_bc1 = (h->t_dev || no_t) ? 0.0f : inv_bias_correction(cfg.beta1, t);
    st.inv_bc2 = (fused && !h->t_dev) ? inv_bias_correction(h->upd_beta2, t) : 0.0f;
    st.t_dev = no_t ? nullptr : h->t_dev;
    st.lr_dev = h->lr_dev;
    st.beta1 = cfg.beta1;
    st.beta2 = fused ? h->upd_beta2 : 0.0f;
    // A small whole step runs its task-space pass, label scan included, as one
    // cluster launch after the logits (the forward reads no label).
    const bool small = part == kStepFull && h->own_out.empty() && task_small_usable(n, V, dm, cf32);
    // A small fp32 MLP classifier (the tiny configurations: a few dozen rows,
    // at most two Linear layers) runs its whole step in one CTA.
    if (part == kStepFull && !h->bf16 && !gh && h->own_out.empty() && h->dx_in == nullptr &&
        h->lw.size() <= static_cast<size_t>(kTinyStepMaxLayers)) {
        bool lin = true;
        for (const LayerWs& L : h->lw) lin = lin && (L.kind == BOM_LAYER_LINEAR || L.kind == BOM_LAYER_LINEAR_GELU);
        TinyStepArgs ta{};
        const int nl = static_cast<int>(h->lw.size());
        int dim[kTinyStepMaxLayers + 2] = {};
        bool bias[kTinyStepMaxLayers + 1] = {};
        dim[0] = static_cast<int>(cfg.d_in);
        for (int k = 0; k < nl; ++k) {
            dim[k + 1] = static_cast<int>(h->lw[k].d_out);
            bias[k] = h->lw[k].bias;
        }
        dim[nl + 1] = static_cast<int>(V);
        bias[nl] = cfg.head_bias != 0;
        if (lin && cfg.d_in <= kTinyStepMaxWidth && V <= kTinyStepMaxWidth &&
            tiny_step_layout(static_cast<int>(n), nl, dim, bias, &ta.lay)) {
            ta.x = static_cast<const float*>(x);
            ta.labels = labels;
            ta.n = static_cast<int>(n);
            ta.nl = nl;
            for (int k = 0; k <= nl + 1; ++k) ta.dim[k] = dim[k];
            int pt = 0;
            for (int k = 0; k <= nl; ++k) {
                if (k < nl) ta.gelu[k] = h->lw[k].kind == BOM_LAYER_LINEAR_GELU ? 1 : 0;
                ta.tw[k] = pt;
                ta.W[k] = static_cast<const float*>(params[pt++]);
                ta.tb[k] = bias[k] ? pt : -1;
                ta.b[k] = bias[k] ? static_cast<const float*>(params[pt++]) : nullptr;
            }
            for (int t2 = 0; t2 < pt; ++t2) {
                ta.u[t2] = fused ? nullptr : static_cast<float*>(grads[t2]);
                ta.theta[t2] = fused ? h->upd_theta[t2] : nullptr;
                ta.v[t2] = fused ? h->upd_v[t2] : nullptr;
                ta.wd[t2] = fused ? h->upd_wd[t2] : 0.0f;
                ta.copy[t2] = static_cast<float*>(params[t2]);
            }
            ta.ignore = cfg.ignore_index;
            ta.lambda = cfg.lambda;
            ta.beta1 = cfg.beta1;
            ta.q = q;
            ta.qhat_out = h->qhat;
            ta.s_out = h->s;
            ta.lse_out = h->lse;
            ta.beta2 = fused ? h->upd_beta2 : 0.0f;
            ta.eps = fused ? h->upd_eps : 0.0f;
            ta.st = st;
            ta.sc = h->sc;
            ta.t_adv = h->t_dev;
            if (cudaMemsetAsync(&h->sc->status, 0, sizeof(int32_t), s) != cudaSuccess) return BOM_ECUDA;
            double fl = 0.0;
            for (int k = 0; k <= nl; ++k) fl += 6.0 * n * dim[k] * dim[k + 1];
            BOM_TRY(traced(h, s, "tiny_step", fl, 4.0 * (n * dim[0] + 3.0 * ta.lay.floats),
                           [&] { return launch_tiny_step(ta, s); }));
            return cudaPeekAtLastError() == cudaSuccess ? BOM_OK : BOM_ECUDA;
        }
    }
    if (first_part) {   // later parts keep the status word of the first
        if (cudaMemsetAsync(&h->sc->status, 0, sizeof(int32_t), s) != cudaSuccess) return BOM_ECUDA;
        // a vocabulary shard checks labels against the whole vocabulary
        if (!small)
            BOM_TRACED("labels_scan", 0, 4.0 * n,
                       launch_labels_scan(labels, n, vshard ? h->vs_total : V, cfg.ignore_index, cfg.lambda, st,
                                          h->sc, s, shard));
    }

    // ---------------------------------------------------------------- forward
    // (the second half of a sharded step finds the activations, R and the
    // residual pass's column partials of its rows in the workspace)
    const bool run_fwd = first_part;
    const void* xin = x;
    int pi = 0;
    std::vector<int> pidx(h->lw.size());
    for (size_t l = 0; l < h->lw.size(); ++l) {
        LayerWs& L = h->lw[l];
        pidx[l] = pi;
        if (!run_fwd) {
            pi += L.kind == BOM_LAYER_SWIGLU ? 3 : (L.kind == BOM_LAYER_RMSNORM ? 1 : (L.bias ? 2 : 1));
            xin = L.out;
            continue;
        }
        if (L.kind == BOM_LAYER_SWIGLU) {
            const void* Wg = params[pi];
            const void* Wu = params[pi + 1];
            const void* Wd = params[pi + 2];
            pi += 3;
            const int64_t d = L.d_in, f = L.d_out;
            GemmDesc g = gemm1(n, f, d, kmaj(xin, d), kmaj(Wg, d));
            g.B[1] = kmaj(Wu, d);
            g.dual_b = true;
            g.epi_kind = EPI_SWIGLU_FWD;
            g.epi.out = L.A;
            g.epi.ld_out = f;
            g.epi.out2 = L.G;
            g.epi.ld_out2 = L.gu_ld;
            BOM_TRY(run_gemm(h, g, s));
            GemmDesc g2 = gemm1(n, d, f, kmaj(L.A, f), kmaj(Wd, f));
            g2.epi.resid = xin;
            g2.epi.ld_resid = d;
            g2.epi.out = L.out;
            g2.epi.ld_out = d;
            BOM_TRY(run_gemm(h, g2, s));
        } else if (L.kind == BOM_LAYER_RMSNORM) {
            const void* gamma = params[pi++];
            BOM_TRACED("rmsnorm_fwd", 4.0 * n * L.d_in, 2.0 * h->esz * n * L.d_in + 4.0 * n,
                       launch_rmsnorm_fwd(xin, gamma, L.out, L.rstd, n, L.d_in, cf32, h->sc, s));
        } else {
            const void* W = params[pi++];
            const void* b = L.bias ? params[pi++] : nullptr;
            GemmDesc g = gemm1(n, L.d_out, L.d_in, kmaj(xin, L.d_in), kmaj(W, L.d_in));
            g.epi.bias = b;
            g.epi.out = L.out;
            g.epi.ld_out = L.d_out;
            g.epi.out_f32 = cf32;
            if (L.kind == BOM_LAYER_LINEAR_GELU) {
                g.epi.act = ACT_GELU;
                g.epi.out2 = L.pre;
                g.epi.ld_out2 = L.d_out;
                g.epi.out2_f32 = cf32;
            }
            BOM_TRY(run_gemm(h, g, s));
        }
        xin = L.out;
    }
    const int head_w = pi;
    const void* Wh = params[pi++];
    const int head_b = cfg.head_bias ? pi++ : -1;
    const void* bh = head_b >= 0 ? params[head_b] : nullptr;
    if (run_fwd) {
        GemmDesc g = gemm1(n, V, dm, kmaj(xin, dm), kmaj(Wh, dm));
        // the small task pass forms the row statistics from Z itself: on the
        // tensor-core engine its logits are a plain linear GEMM (narrow tiles
        // when there are few), without the per-tile softmax statistics
        g.epi_kind = small && h->bf16 ? EPI_LINEAR : EPI_LOGITS;
        g.epi.bias = bh;
        g.epi.out = h->Z;
        g.epi.ld_out = h->ldz;
        g.epi.out_f32 = cf32;
        if (g.epi_kind == EPI_LOGITS) {
            g.epi.stats = h->stats;
            g.epi.ld_stats = h->ntiles;
        }
        BOM_TRY(run_gemm(h, g, s));
    }
    if (run_fwd && !h->bf16 && !small)
        BOM_TRACED("row_stats_f32", 0, 4.0 * n * V,
                   launch_row_stats_f32(static_cast<const float*>(h->Z), h->ldz, n, V, h->stats, h->sc, s));

    // ---------------------------------------------------------------- task space
    const bool own = !h->own_out.empty();
    // with one u pass the small task pass also writes the head bias numerator
    const bool small_bias = small && !gh && head_b >= 0;
    if (small) {
        void* hb = small_bias ? (fused ? static_cast<void*>(uvec(head_b)) : grads[head_b]) : nullptr;
        BOM_TRY(traced(h, s, "task_small", 2.0 * V * dm,
                       2.0 * h->esz * n * h->ldz + h->esz * (n + V) * dm + 12.0 * V, [&] {
                           return launch_task_small(h->Z, cf32, h->ldz, labels, n, V, cfg.ignore_index, cfg.lambda,
                                                    cfg.beta1, xin, Wh, dm, q, h->s, h->qhat, h->lse, h->cvec,
                                                    h->wvec, hb, fused ? 1 : cf32, 1.0f - cfg.lambda, cfg.lambda, st,
                                                    h->sc, s);
                       }));
    }
    if (part == kVBegin) {   // this shard's part of each row's log-sum-exp, for the caller's exchange
        BOM_TRACED("lse_part", 0, 8.0 * n * h->ntiles + 4.0 * n,
                   launch_vshard_lse_part(h->stats, h->ntiles, n, vio->lse_part, h->sc, s));
        return cudaPeekAtLastError() == cudaSuccess ? BOM_OK : BOM_ECUDA;
    }
    if (part == kVMid) {
        // the row log-sum-exp from every shard's part, then R over this shard's
        // columns (the label of column j is vs_first + j)
        BOM_TRACED("row_lse", 0, 4.0 * vio->nsh * n + 12.0 * n,
                   launch_vshard_lse(vio->lse_parts, vio->nsh, n, h->Z, cf32, h->ldz, h->vs_first, V, labels,
                                     cfg.ignore_index, h->lse, h->ce, st, h->sc, s));
        BOM_TRACED("residual", 0, 2.0 * h->esz * n * h->ldz + 4.0 * resid_blocks(n) * V + 8.0 * n,
                   launch_residual(h->Z, cf32, h->ldz, n, V, h->lse, labels, cfg.ignore_index, h->colpart, h->sc, s,
                                   h->vs_first));
    }
    if (run_fwd && !small) {
        BOM_TRACED("row_lse", 0, 8.0 * n * h->ntiles + 12.0 * n,
                   launch_row_lse(h->Z, cf32, h->ldz, n, V, h->stats, h->ntiles, labels, cfg.ignore_index, h->lse,
                                  h->ce, h->sc, s));
        // residual pass: reads and rewrites Z once, writes the column partial sums
        BOM_TRACED("residual", 0, 2.0 * h->esz * n * h->ldz + 4.0 * resid_blocks(n) * V + 8.0 * n,
                   launch_residual(h->Z, cf32, h->ldz, n, V, h->lse, labels, cfg.ignore_index, h->colpart, h->sc,
                                   s));
    }
    if (part == kShardBegin) {   // this shard's sums, for the caller's exchange
        BOM_TRACED("shard_sums", 0, 4.0 * resid_blocks(n) * V + 4.0 * n + 8.0 * (V + 3),
                   launch_shard_sums(h->colpart, resid_blocks(n), h->ce, n, V, xch_out, h->sc, s));
        return cudaPeekAtLastError() == cudaSuccess ? BOM_OK : BOM_ECUDA;
    }
    if (part == kShardEnd) {
        BOM_TRACED("shard_scalars", 0, 8.0 * 3, launch_shard_scalars_in(xch_in, V, cfg.lambda, st, h->sc, s));
        BOM_TRACED("finish_sq", 0, 4.0 * resid_blocks(n) * V + 8.0 * V + 24.0 * V,
                   launch_shard_finish_sq(xch_in, h->colpart, resid_blocks(n), V, cfg.beta1, q, h->s, h->qhat,
                                          h->sshard, h->sc, s));
    } else if (!small && part != kVEnd) {
        BOM_TRACED("finish_sq", 0, 4.0 * resid_blocks(n) * V + 20.0 * V,
                   launch_finish_sq(h->colpart, resid_blocks(n), V, cfg.beta1, q, h->s, h->qhat, h->sc, s));
    }
    if (own)   // per-row residual norms for the cancellation ratio
        BOM_TRACED("row_norm", 2.0 * n * V, h->esz * n * h->ldz + 4.0 * n,
                   launch_row_norm(h->Z, cf32, h->ldz, n, V, h->rnorm, h->sc, s));
    if (!small && part != kVEnd) {
        // (a row-sharded step's loss comes from the shards' summed CE; a
        // vocabulary shard's is its part of the batch's)
        BOM_TRACED("scalars", 0, 4.0 * (n + V),
                   launch_scalars(shard ? nullptr : h->ce, n, h->s, V, own ? h->rnorm : nullptr, h->sc, s));
        // c = colsum_{I_t}(H) and w = W^T qhat (the rank-1 / broadcast factors of the reprojection)
        BOM_TRACED("colsum", 2.0 * n * dm, h->esz * n * dm,
                   launch_colsum(xin, cf32, dm, n, dm, labels, cfg.ignore_index, nullptr, 1.0f, h->part, h->cvec,
                                 1, h->sc, s));
        BOM_TRACED("colsum", 2.0 * V * dm, h->esz * V * dm,
                   launch_colsum(Wh, cf32, dm, V, dm, nullptr, 0, h->qhat, 1.0f, h->part, h->wvec, 1, h->sc, s));
    }
    if (own)
        BOM_TRACED("colsum", 2.0 * V * dm, h->esz * V * dm,
                   launch_colsum(Wh, cf32, dm, V, dm, nullptr, 0, h->s, 1.0f, h->part, h->wsvec, 1, h->sc, s));

    // ---------------------------------------------------------------- backward
    // passes: 0 = u, 1 = g, 2 = h = Jbar^T qhat, 3 = own-step projection Jbar^T s_t.
    // Within the head and every layer the input cotangent is formed before the
    // weight gradients: a fused update rewrites the compute copy of a weight,
    // so it runs after the last read of that weight in the step.
    int passes[3], npass = 0;
    passes[npass++] = gh ? 1 : 0;
    if (gh) passes[npass++] = 2;
    if (own) passes[npass++] = 3;
    // the fused update takes lr and 1/(1 - beta2^t) from the step scalars
    // the GEMM producing u of tensor k updates it in its epilogue
    // A small bf16 step updates the weights of a grouped weight-gradient
    // launch in its epilogue too (narrow 128 x 64 tiles, one row per lane):
    // only the other tensors' u goes through the scratch to the final update.
    std::vector<char> upd_in_gemm(upd_sep ? bom_param_count(&cfg) : 0, 0);
    auto fuse = [&](GemmDesc& g, int k, bool grouped) {
        if (upd_sep && !(h->bf16 && grouped)) {   // u to the scratch; the update runs after the pass
            g.epi.out = h->uscr + h->uoff[k];
            g.epi.out_f32 = 1;
            return;
        }
        if (upd_sep) upd_in_gemm[k] = 1;
        g.epi.upd_theta = h->upd_theta[k];
        g.epi.upd_v = h->upd_v[k];
        g.epi.upd_wd = h->upd_wd[k];
        g.epi.upd_beta2 = h->upd_beta2;
        g.epi.upd_1mb2 = 1.0f - h->upd_beta2;
        g.epi.upd_eps = h->upd_eps;
        g.epi.out = params[k];   // the compute copy of the updated weight
        g.epi.out_f32 = cf32;
        if (h->bf16) g.epi_kind = EPI_UPDATE;   // tcgen05 path: the update epilogue, one row per lane
    };
    // a vector tensor k whose u is in ubuf (fp32): update it and its compute copy
    auto update_small = [&](int k, int64_t cnt) -> int {
        int r = launch_update(h->upd_theta[k], h->ubuf, 0, nullptr, h->upd_v[k],
                              h->bf16 ? static_cast<uint16_t*>(params[k]) : nullptr, cnt, h->upd_lr, h->upd_wd[k],
                              0.0f, h->upd_beta2, h->upd_eps, 0.0f, nullptr, 0.0f, h->sc, s, true);
        if (r == BOM_OK && !h->bf16 &&
            cudaMemcpyAsync(params[k], h->upd_theta[k], cnt * 4, cudaMemcpyDeviceToDevice, s) != cudaSuccess)
            r = BOM_ECUDA;
        return r;
    };
    for (int pp = 0; pp < npass; ++pp) {
        const int pass = passes[pp];
        void* const* outp = pass == 3 ? h->own_out.data() : (pass == 2 ? h_out : grads);
        const int of32 = pass >= 2 ? 1 : cf32;
        const float* cr = &h->sc->coef_r[pass];
        const float* cq = &h->sc->coef_q[pass];
        const int64_t kfull = pass >= 2 ? 0 : 1;  // the h and own-step passes have no residual term
        const float* tvec = pass == 3 ? h->s : h->qhat;      // broadcast task-space vector
        const float* wtvec = pass == 3 ? h->wsvec : h->wvec; // W^T of it
        // the cotangent of X goes out with the u (or g) pass when requested
        const bool want_dx = h->dx_in != nullptr && pass < 2;
        int cur = 0;
        void* const dh_dst = h->lw.empty() ? h->dx_in : h->dx[cur];
        if ((!h->lw.empty() || want_dx) && part == kVEnd) {
            // the head's input cotangent: the vocabulary shards' parts summed by
            // the caller, in the compute dtype
            BOM_TRACED("cast", 0, (4.0 + h->esz) * n * dm, launch_cast_f32(vio->dh_sum, dh_dst, n * dm, cf32, h->sc, s));
        } else if (!h->lw.empty() || want_dx) {   // head input: a R W + b 1_{I_t} w^T  (times GELU' of the last layer)
            GemmDesc g = gemm1(n, dm, kfull * V, kmaj(h->Z, h->ldz), mnmaj(Wh, dm));
            g.epi.alpha_dev = cr;
            g.epi.beta_dev = cq;
            g.epi.bw = wtvec;
            g.epi.mask_labels = labels;
            g.epi.ignore_index = cfg.ignore_index;
            if (!h->lw.empty() && h->lw.back().kind == BOM_LAYER_LINEAR_GELU) {
                g.epi.act = ACT_DGELU;
                g.epi.aux = h->lw.back().pre;
                g.epi.ld_aux = h->lw.back().d_out;
            }
            // a vocabulary shard's part goes to the caller in fp32, for the sum
            // over shards (the GELU' factor distributes over it)
            g.epi.out = part == kVMid ? static_cast<void*>(vio->dh_part) : dh_dst;
            g.epi.ld_out = dm;
            g.epi.out_f32 = part == kVMid ? 1 : cf32;
            if (cs_fused && !h->lw.empty() && h->lw.back().cspart != nullptr) {
                g.epi.colsum = h->lw.back().cspart;
                g.epi.ld_colsum = h->lw.back().d_out;
                cs_ready.back() = 1;
            }
            BOM_TRY(run_gemm(h, g, s));
        }
        // The head weight gradient contracts over the same n rows as the
        // sublayers' weight gradients: with a SwiGLU first layer it waits and
        // runs in one launch with that layer's (every operand stays live), and
        // so do a SwiGLU second layer's.  One work list over all of them
        // leaves one partial wave instead of one per launch.
        GemmDesc head_dw;
        GemmDesc pend[3];
        int npend = 0;
        // Up to two Linear layers in front of the head: their cotangents stay in
        // dx[0] and dx[1] until the pass ends, so their weight gradients and
        // the head's can run as one grouped launch after the last input
        // cotangent (every weight is still read before its fused update).
        // (a vocabulary shard's head weight gradient runs in its middle part,
        // the backbone's in its last)
        bool defer_lin = !vshard && kfull == 1 && !h->lw.empty() && h->lw.size() <= 2;
        for (const LayerWs& L : h->lw)
            defer_lin = defer_lin && (L.kind == BOM_LAYER_LINEAR || L.kind == BOM_LAYER_LINEAR_GELU);
        const bool defer_head =
            (!vshard && h->bf16 && kfull == 1 && !h->lw.empty() && h->lw[0].kind == BOM_LAYER_SWIGLU) || defer_lin;
        if (part != kVEnd) {   // head weight: a R^T H + b qhat (x) c
            GemmDesc g = gemm1(V, dm, kfull * n, mnmaj(h->Z, h->ldz), mnmaj(xin, dm));
            g.epi.alpha_const = 1.0f;
            g.epi.alpha_dev = cr;
            g.epi.beta_dev = cq;
            g.epi.r1u = tvec;
            g.epi.r1v = h->cvec;
            g.epi.out = fused ? nullptr : outp[head_w];
            g.epi.ld_out = dm;
            g.epi.out_f32 = of32;
            if (fused) fuse(g, head_w, defer_head);
            if (defer_head)
                head_dw = g;
            else
                BOM_TRY(run_gemm(h, g, s));
        }
        if (head_b >= 0 && part != kVEnd) {
            const float a = pass == 0 ? 1.0f - cfg.lambda : (pass == 1 || pass == 3 ? 1.0f : 0.0f);
            const float b = pass == 0 ? cfg.lambda : (pass == 2 ? 1.0f : 0.0f);
            if (shard)   // this shard's share: a s^shard + b (N_t^shard / N_t) qhat
                BOM_TRACED("axpby", 3.0 * V, 12.0 * V,
                           launch_shard_bias(h->sshard, h->qhat, a, b, V, outp[head_b], of32, h->sc, s));
            else if (small_bias)
                ;   // written by the small task pass
            else
                BOM_TRACED("axpby", 3.0 * V, 12.0 * V,
                           launch_axpby(h->s, h->qhat, a, b, V, fused ? uvec(head_b) : outp[head_b], fused ? 1 : of32,
                                        h->sc, s));
            if (fused && !upd_sep) BOM_TRY(update_small(head_b, V));
        }
        // a vocabulary shard's middle part ends with its head: the backbone
        // waits for the caller's sum of the input cotangent's parts
        if (part == kVMid) return cudaPeekAtLastError() == cudaSuccess ? BOM_OK : BOM_ECUDA;
        for (int l = static_cast<int>(h->lw.size()) - 1; l >= 0; --l) {
            const LayerWs& L = h->lw[l];
            const void* xl = l == 0 ? x : h->lw[l - 1].out;
            const void* dcur = h->dx[cur];
            const int p0 = pidx[l];
            const LayerWs* prev = l > 0 ? &h->lw[l - 1] : nullptr;
            const bool dx_next = prev != nullptr || want_dx;
            void* const dxo = prev ? h->dx[cur ^ 1] : h->dx_in;
            if (L.kind == BOM_LAYER_SWIGLU) {
                const int64_t d = L.d_in, f = L.d_out;
                const void* Wg = params[p0];
                const void* Wu = params[p0 + 1];
                const void* Wd = params[p0 + 2];
                // the second sublayer's weight gradients wait for the first's launch:
                // its dy (dx[cur]) is not written again, the first layer's input
                // gradient goes to the caller's buffer
                const bool defer_w = defer_head && l == 1 && h->dG2 != nullptr;
                void* const dGl = defer_w ? h->dG2 : h->dG;
                void* const dUl = defer_w ? h->dU2 : h->dU;
                {   // dA = dy W_d, then dG = dA u SiLU'(g), dU = dA SiLU(g)
                    GemmDesc g = gemm1(n, f, d, kmaj(dcur, d), mnmaj(Wd, f));
                    g.epi_kind = EPI_SWIGLU_BWD;
                    g.epi.aux = L.G;
                    g.epi.ld_aux = L.gu_ld;
                    g.epi.out = dGl;
                    g.epi.ld_out = f;
                    g.epi.out2 = dUl;
                    g.epi.ld_out2 = f;
                    BOM_TRY(run_gemm(h, g, s));
                }
                if (dx_next) {   // dx = dy + dG W_g + dU W_u
                    GemmDesc g = gemm1(n, d, f, kmaj(dGl, f), mnmaj(Wg, d));
                    g.nseg = 2;
                    g.A[1] = kmaj(dUl, f);
                    g.B[1] = mnmaj(Wu, d);
                    g.K[1] = f;
                    g.epi.resid = dcur;
                    g.epi.ld_resid = d;
                    if (prev && prev->kind == BOM_LAYER_LINEAR_GELU) {
                        g.epi.act = ACT_DGELU;
                        g.epi.aux = prev->pre;
                        g.epi.ld_aux = prev->d_out;
                    }
                    g.epi.out = dxo;
                    g.epi.ld_out = d;
                    g.epi.out_f32 = cf32;
                    if (cs_fused && prev && prev->cspart != nullptr) {
                        g.epi.colsum = prev->cspart;
                        g.epi.ld_colsum = prev->d_out;
                        cs_ready[l - 1] = 1;
                    }
                    BOM_TRY(run_gemm(h, g, s));
                }
                {   // dW_g = dG^T x, dW_u = dU^T x, dW_d = dy^T A: one launch over their tiles
                    GemmDesc gw[7];
                    gw[0] = gemm1(f, d, n, mnmaj(dGl, f), mnmaj(xl, d));
                    gw[1] = gemm1(f, d, n, mnmaj(dUl, f), mnmaj(xl, d));
                    gw[2] = gemm1(d, f, n, mnmaj(dcur, d), mnmaj(L.A, f));
                    const int pk[3] = {p0, p0 + 1, p0 + 2};
                    for (int i = 0; i < 3; ++i) {
                        gw[i].epi.out = fused ? nullptr : outp[pk[i]];
                        gw[i].epi.ld_out = i < 2 ? d : f;
                        gw[i].epi.out_f32 = of32;
                        if (fused) fuse(gw[i], pk[i], true);
                    }
                    if (defer_w) {
                        for (int i = 0; i < 3; ++i) pend[npend++] = gw[i];
                    } else {
                        int ng = 3;
                        if (defer_head && l == 0) {   // the second sublayer's and the head's, deferred
                            for (int i = 0; i < npend; ++i) gw[ng++] = pend[i];
                            gw[ng++] = head_dw;
                        }
                        BOM_TRY(run_gemm_group(h, gw, ng, s));
                    }
                }
            } else if (L.kind == BOM_LAYER_RMSNORM) {
                const int64_t d = L.d_in;
                const void* gamma = params[p0];
                // dgamma_j = sum_i rstd_i dy_ij x_ij
                BOM_TRACED("colsum", 3.0 * n * d, 2.0 * h->esz * n * d,
                           launch_colsum2(dcur, xl, cf32, d, n, d, nullptr, 0, L.rstd, 1.0f, h->part,
                                          fused ? uvec(p0) : outp[p0], fused ? 1 : of32, h->sc, s));
                if (dx_next) {
                    const void* pre = (prev && prev->kind == BOM_LAYER_LINEAR_GELU) ? prev->pre : nullptr;
                    BOM_TRACED("rmsnorm_bwd", 8.0 * n * d, 3.0 * h->esz * n * d + 4.0 * n,
                               launch_rmsnorm_bwd(dcur, xl, gamma, L.rstd, pre, dxo, n, d, cf32, h->sc, s));
                }
                if (fused && !upd_sep) BOM_TRY(update_small(p0, d));   // after the last read of gamma
            } else {
                const void* W = params[p0];
                if (dx_next) {   // dx = dPre W (times GELU' of the previous layer)
                    GemmDesc g = gemm1(n, L.d_in, L.d_out, kmaj(dcur, L.d_out), mnmaj(W, L.d_in));
                    if (prev && prev->kind == BOM_LAYER_LINEAR_GELU) {
                        g.epi.act = ACT_DGELU;
                        g.epi.aux = prev->pre;
                        g.epi.ld_aux = prev->d_out;
                    }
                    g.epi.out = dxo;
                    g.epi.ld_out = L.d_in;
                    g.epi.out_f32 = cf32;
                    if (cs_fused && prev && prev->cspart != nullptr) {
                        g.epi.colsum = prev->cspart;
                        g.epi.ld_colsum = prev->d_out;
                        cs_ready[l - 1] = 1;
                    }
                    BOM_TRY(run_gemm(h, g, s));
                }
                {   // dW = dPre^T x
                    GemmDesc g = gemm1(L.d_out, L.d_in, n, mnmaj(dcur, L.d_out), mnmaj(xl, L.d_in));
                    g.epi.out = fused ? nullptr : outp[p0];
                    g.epi.ld_out = L.d_in;
                    g.epi.out_f32 = of32;
                    if (fused) fuse(g, p0, defer_lin);
                    if (defer_lin) {
                        pend[npend++] = g;
                        if (l == 0) {   // the last layer of the pass: these and the head's, one launch
                            GemmDesc gw[3];
                            int ng = 0;
                            for (int i = 0; i < npend; ++i) gw[ng++] = pend[i];
                            gw[ng++] = head_dw;
                            BOM_TRY(run_gemm_group(h, gw, ng, s));
                        }
                    } else {
                        BOM_TRY(run_gemm(h, g, s));
                    }
                }
                if (L.bias && fold_bias) {
                    usrc[p0 + 1] = dcur;   // its column sum over the n rows is u of the bias
                } else if (L.bias && cs_ready[l]) {
                    usrc[p0 + 1] = L.cspart;   // u of the bias: the sum of the block column sums
                    urows[p0 + 1] = (n + 31) / 32;
                    usf32[p0 + 1] = 1;
                } else if (L.bias) {
                    BOM_TRACED("colsum", 2.0 * n * L.d_out, h->esz * n * L.d_out,
                               launch_colsum(dcur, cf32, L.d_out, n, L.d_out, nullptr, 0, nullptr, 1.0f, h->part,
                                             fused ? uvec(p0 + 1) : outp[p0 + 1], fused ? 1 : of32, h->sc, s));
                    if (fused && !upd_sep) BOM_TRY(update_small(p0 + 1, L.d_out));
                }
            }
            if (dx_next) cur ^= 1;
        }
    }
    bool advanced = false;
    if (upd_sep) {   // the other tensors' BOM-AdamW update, after their last read in the step
        const int np = bom_param_count(&cfg);
        std::vector<float*> th, vv;
        std::vector<const float*> uu;
        std::vector<void*> cp;
        std::vector<int64_t> nn, rr;
        std::vector<float> wd;
        std::vector<const void*> src;
        std::vector<int> sf;
        int64_t tot = 0;
        for (int k = 0; k < np; ++k) {
            if (upd_in_gemm[k]) continue;
            th.push_back(h->upd_theta[k]);
            vv.push_back(h->upd_v[k]);
            uu.push_back(h->uscr + h->uoff[k]);
            cp.push_back(params[k]);
            nn.push_back(h->unum[k]);
            wd.push_back(h->upd_wd[k]);
            src.push_back(usrc.empty() ? nullptr : usrc[k]);
            rr.push_back(urows.empty() ? 0 : urows[k]);
            sf.push_back(usf32.empty() ? cf32 : usf32[k]);
            tot += h->unum[k];
        }
        if (!th.empty()) {
            BOM_TRY(traced(h, s, "update", 0, 22.0 * tot, [&] {
                return launch_update_multi(static_cast<int>(th.size()), th.data(), vv.data(), uu.data(), cp.data(),
                                           cf32, nn.data(), wd.data(), src.data(), rr.data(), sf.data(),
                                           h->upd_beta2, h->upd_eps, h->sc, h->t_dev, s);
            }));
            advanced = true;   // the update of a small step advances the device step counter itself
        }
    }
    if (h->t_dev && !advanced) launch_advance_step(h->t_dev, h->sc, s);
#undef BOM_TRY
    return cudaPeekAtLastError() == cudaSuccess ? BOM_OK : BOM_ECUDA;
}

}  // namespace

extern "C" {

bom_status bom_step(bom_handle* h, const void* x, const int32_t* labels, int64_t n, void* const* params, float* q,
                    int64_t t, void* const* grads, void* const* h_out, void* stream) {
    const bom_status rc = check_step_args(h, x, labels, n, params, q, t, grads, h_out, kStepFull);
    if (rc != BOM_OK) return rc;
    const NvtxRange nvtx_step("bom_step");
    return step_impl(h, x, labels, n, params, q, t, grads, h_out, stream, kStepFull, nullptr, nullptr);
}

bom_status bom_step_shard_begin(bom_handle* h, const void* x, const int32_t* labels, int64_t n_rows,
                                void* const* params, double* xch, void* stream) {
    const bom_status rc = check_step_args(h, x, labels, n_rows, params, nullptr, 1, nullptr, nullptr, kShardBegin);
    if (rc != BOM_OK) return rc;
    if (!xch) return BOM_EINVAL;
    if ((reinterpret_cast<uintptr_t>(xch) & 7u) != 0) return BOM_ENOTSUP;
    const NvtxRange nvtx_step("bom_step_shard_begin");
    return step_impl(h, x, labels, n_rows, params, nullptr, 1, nullptr, nullptr, stream, kShardBegin, xch, nullptr);
}

bom_status bom_step_shard_end(bom_handle* h, const void* x, const int32_t* labels, int64_t n_rows,
                              void* const* params, float* q, int64_t t, const double* xch, void* const* grads,
                              void* const* h_out, void* stream) {
    const bom_status rc = check_step_args(h, x, labels, n_rows, params, q, t, grads, h_out, kShardEnd);
    if (rc != BOM_OK) return rc;
    if (!xch || n_rows != h->shard_n) return BOM_EINVAL;   // no matching first half
    if ((reinterpret_cast<uintptr_t>(xch) & 7u) != 0) return BOM_ENOTSUP;
    const NvtxRange nvtx_step("bom_step_shard_end");
    return step_impl(h, x, labels, n_rows, params, q, t, grads, h_out, stream, kShardEnd, nullptr, xch);
}

bom_status bom_step_vshard_begin(bom_handle* h, const void* x, const int32_t* labels, int64_t n_rows,
                                 void* const* params, int64_t v_total, int64_t v_first, float* lse_part,
                                 void* stream) {
    bom_status rc = check_step_args(h, x, labels, n_rows, params, nullptr, 1, nullptr, nullptr, kVBegin);
    if (rc != BOM_OK) return rc;
    if (!lse_part || v_total < 1 || v_total > INT32_MAX || v_first < 0 || v_first > v_total - h->cfg.d_out)
        return BOM_EINVAL;
    if ((reinterpret_cast<uintptr_t>(lse_part) & 3u) != 0) return BOM_ENOTSUP;
    const NvtxRange nvtx_step("bom_step_vshard_begin");
    h->vs_stage = 0;
    h->vs_total = v_total;
    h->vs_first = v_first;
    VShardIo io;
    io.lse_part = lse_part;
    rc = step_impl(h, x, labels, n_rows, params, nullptr, 1, nullptr, nullptr, stream, kVBegin, nullptr, nullptr, &io);
    if (rc == BOM_OK) {
        h->vs_n = n_rows;
        h->vs_stage = 1;
    }
    return rc;
}

bom_status bom_step_vshard_mid(bom_handle* h, const void* x, const int32_t* labels, int64_t n_rows,
                               void* const* params, float* q, int64_t t, const float* lse_parts, int32_t n_shards,
                               void* const* grads, float* dh_part, void* stream) {
    bom_status rc = check_step_args(h, x, labels, n_rows, params, q, t, grads, nullptr, kVMid);
    if (rc != BOM_OK) return rc;
    if (h->vs_stage != 1 || n_rows != h->vs_n) return BOM_EINVAL;   // no matching first part
    if (!lse_parts || n_shards < 1 || n_shards > kMaxVocabShards) return BOM_EINVAL;
    if ((reinterpret_cast<uintptr_t>(lse_parts) & 3u) != 0) return BOM_ENOTSUP;
    const bool need_dh = !h->lw.empty() || h->dx_in != nullptr;
    if (need_dh && !dh_part) return BOM_EINVAL;
    if (need_dh && !aligned16(dh_part)) return BOM_ENOTSUP;
    const NvtxRange nvtx_step("bom_step_vshard_mid");
    VShardIo io;
    io.lse_parts = lse_parts;
    io.nsh = n_shards;
    io.dh_part = dh_part;
    h->vs_stage = 0;
    rc = step_impl(h, x, labels, n_rows, params, q, t, grads, nullptr, stream, kVMid, nullptr, nullptr, &io);
    if (rc == BOM_OK) h->vs_stage = 2;
    return rc;
}

bom_status bom_step_vshard_end(bom_handle* h, const void* x, const int32_t* labels, int64_t n_rows,
                               void* const* params, const float* dh_sum, void* const* grads, void* stream) {
    bom_status rc = check_step_args(h, x, labels, n_rows, params, nullptr, 1, grads, nullptr, kVEnd);
    if (rc != BOM_OK) return rc;
    if (h->vs_stage != 2 || n_rows != h->vs_n) return BOM_EINVAL;   // no matching middle part
    const bool need_dh = !h->lw.empty() || h->dx_in != nullptr;
    if (need_dh && !dh_sum) return BOM_EINVAL;
    if (need_dh && !aligned16(dh_sum)) return BOM_ENOTSUP;
    const NvtxRange nvtx_step("bom_step_vshard_end");
    VShardIo io;
    io.dh_sum = dh_sum;
    h->vs_stage = 0;
    return step_impl(h, x, labels, n_rows, params, nullptr, 1, grads, nullptr, stream, kVEnd, nullptr, nullptr, &io);
}

bom_status bom_set_input_grad(bom_handle* h, void* dx) {
    if (!h) return BOM_EINVAL;
    if (dx && !aligned16(dx)) return BOM_ENOTSUP;
    h->dx_in = dx;
    return BOM_OK;
}

bom_status bom_set_own_step_output(bom_handle* h, void* const* o) {
    if (!h) return BOM_EINVAL;
    if (!o) {
        h->own_out.clear();
        return BOM_OK;
    }
    const int np = bom_param_count(&h->cfg);
    std::vector<void*> v(o, o + np);
    for (void* p : v) {
        if (!p) return BOM_EINVAL;
        if (!aligned16(p)) return BOM_ENOTSUP;
    }
    h->own_out = v;
    return BOM_OK;
}

bom_status bom_set_fused_update(bom_handle* h, float* const* theta, float* const* v, const float* wd, float lr,
                                float beta2, float eps) {
    if (!h) return BOM_EINVAL;
    if (!theta) {
        h->fused_upd = false;
        return BOM_OK;
    }
    if (!v || !wd || !(beta2 >= 0.0f && beta2 < 1.0f) || !(eps >= 0.0f)) return BOM_EINVAL;
    const int np = bom_param_count(&h->cfg);
    for (int i = 0; i < np; ++i) {
        if (!theta[i] || !v[i]) return BOM_EINVAL;
        if (!aligned16(theta[i]) || !aligned16(v[i])) return BOM_ENOTSUP;
    }
    h->upd_theta.assign(theta, theta + np);
    h->upd_v.assign(v, v + np);
    h->upd_wd.assign(wd, wd + np);
    h->upd_lr = lr;
    h->upd_beta2 = beta2;
    h->upd_eps = eps;
    h->fused_upd = true;
    return BOM_OK;
}

bom_status bom_set_step_scalars(bom_handle* h, int64_t* t_dev, const float* lr_dev) {
    if (!h) return BOM_EINVAL;
    if ((reinterpret_cast<uintptr_t>(t_dev) & 7u) != 0 || (reinterpret_cast<uintptr_t>(lr_dev) & 3u) != 0)
        return BOM_ENOTSUP;
    h->t_dev = t_dev;
    h->lr_dev = lr_dev;
    return BOM_OK;
}

}  // extern "C"

struct bom_graph {
    cudaGraph_t graph = nullptr;
    cudaGraphExec_t exec = nullptr;
    long long kernels = 0;   // kernel nodes: bom_launch_count advances by this much per launch
};

extern "C" {

bom_status bom_graph_capture(bom_handle* h, const void* x, const int32_t* labels, int64_t n_rows,
                             void* const* params, float* q, void* const* grads, void* const* h_out,
                             bom_graph** out) {
    if (!h || !out) return BOM_EINVAL;
    *out = nullptr;
    if (!h->t_dev || h->tracing) return BOM_EINVAL;
    cudaStream_t cs = nullptr;
    if (cudaStreamCreateWithFlags(&cs, cudaStreamNonBlocking) != cudaSuccess) return BOM_ECUDA;
    // relaxed mode: the first launch of a GEMM shape sets kernel attributes
    // (not stream work) while the capture is open
    if (cudaStreamBeginCapture(cs, cudaStreamCaptureModeRelaxed) != cudaSuccess) {
        cudaStreamDestroy(cs);
        return BOM_ECUDA;
    }
    const long long n0 = bom::g_launches.load();
    const bom_status rc = bom_step(h, x, labels, n_rows, params, q, 0, grads, h_out, cs);
    // the captured launches ran nothing: they are counted when the graph runs
    const long long nk = bom::g_launches.load() - n0;
    bom::g_launches.fetch_sub(nk);
    cudaGraph_t g = nullptr;
    const cudaError_t ec = cudaStreamEndCapture(cs, &g);
    cudaStreamDestroy(cs);
    if (rc != BOM_OK || ec != cudaSuccess || g == nullptr) {
        if (g) cudaGraphDestroy(g);
        cudaGetLastError();
        return rc != BOM_OK ? rc : BOM_ECUDA;
    }
    cudaGraphExec_t ge = nullptr;
    if (cudaGraphInstantiate(&ge, g, 0) != cudaSuccess) {
        cudaGraphDestroy(g);
        cudaGetLastError();
        return BOM_ECUDA;
    }
    bom_graph* G = new (std::nothrow) bom_graph;
    if (!G) {
        cudaGraphExecDestroy(ge);
        cudaGraphDestroy(g);
        return BOM_ENOMEM;
    }
    G->graph = g;
    G->exec = ge;
    G->kernels = nk;
    *out = G;
    return BOM_OK;
}

bom_status bom_graph_launch(bom_graph* g, void* stream) {
    if (!g || !g->exec) return BOM_EINVAL;
    if (cudaGraphLaunch(g->exec, static_cast<cudaStream_t>(stream)) != cudaSuccess) return BOM_ECUDA;
    bom::g_launches.fetch_add(g->kernels);
    return BOM_OK;
}

void bom_graph_destroy(bom_graph* g) {
    if (!g) return;
    if (g->exec) cudaGraphExecDestroy(g->exec);
    if (g->graph) cudaGraphDestroy(g->graph);
    delete g;
}

bom_status bom_own_step_moment(bom_handle* h, float* M, const float* o, const float* hvec, float* mhat, int64_t n,
                               float beta1, int64_t t, double* sums, void* stream) {
    if (!h || n < 0 || t < 1 || !(beta1 >= 0.0f && beta1 < 1.0f)) return BOM_EINVAL;
    if (n == 0) return BOM_OK;
    if (!M || !o || !mhat || (sums && !hvec)) return BOM_EINVAL;
    if (!aligned16(M) || !aligned16(o) || !aligned16(mhat) || (hvec && !aligned16(hvec))) return BOM_ENOTSUP;
    const float inv_bc1 = inv_bias_correction(beta1, t);
    const int nb = own_step_blocks(n, device_sm_count());
    launch_own_step_moment(M, o, hvec, mhat, n, beta1, inv_bc1, h->tel_part, nb, sums,
                           static_cast<cudaStream_t>(stream));
    return cudaPeekAtLastError() == cudaSuccess ? BOM_OK : BOM_ECUDA;
}

int64_t bom_stats_transfer_bytes(void) { return static_cast<int64_t>(kStatsBytes); }

bom_status bom_step_outputs(bom_handle* h, const float** qhat, const float** s, const float** lse) {
    if (!h) return BOM_EINVAL;
    if (qhat) *qhat = h->qhat;
    if (s) *s = h->s;
    if (lse) *lse = h->lse;
    return BOM_OK;
}

bom_status bom_stats_decode(const void* src, bom_stats* out) {
    if (!src || !out) return BOM_EINVAL;
    DevScalars sc;
    memcpy(&sc, src, kStatsBytes);
    out->loss = sc.loss;
    out->n_t = sc.n_t;
    out->status = sc.status;
    out->s_norm = sc.s_norm;
    out->r_norm_mean = sc.r_norm_mean;
    out->cancel = sc.r_norm_mean > 0.0f ? sc.s_norm / sc.r_norm_mean : 0.0f;
    return static_cast<bom_status>(sc.status);
}

bom_status bom_get_stats_async(bom_handle* h, void* dst, void* stream) {
    if (!h || !dst) return BOM_EINVAL;
    return cudaMemcpyAsync(dst, h->sc, kStatsBytes, cudaMemcpyDeviceToHost, static_cast<cudaStream_t>(stream)) ==
                   cudaSuccess
               ? BOM_OK
               : BOM_ECUDA;
}

bom_status bom_get_stats(bom_handle* h, bom_stats* out, void* stream) {
    if (!h || !out) return BOM_EINVAL;
    if (cudaStreamSynchronize(static_cast<cudaStream_t>(stream)) != cudaSuccess) return BOM_ECUDA;
    DevScalars sc;
    if (cudaMemcpy(&sc, h->sc, kStatsBytes, cudaMemcpyDeviceToHost) != cudaSuccess) return BOM_ECUDA;
    out->loss = sc.loss;
    out->n_t = sc.n_t;
    out->status = sc.status;
    out->s_norm = sc.s_norm;
    out->r_norm_mean = sc.r_norm_mean;
    out->cancel = sc.r_norm_mean > 0.0f ? sc.s_norm / sc.r_norm_mean : 0.0f;
    return static_cast<bom_status>(sc.status);
}

bom_status bom_update(float* theta, const void* g, int32_t g_dtype, const float* hvec, float* v, uint16_t* theta_bf16,
                      int64_t n, float lr, float wd, float lambda, float beta2, float eps, int64_t t, void* stream) {
    if (n < 0 || t < 1) return BOM_EINVAL;
    if (n == 0) return BOM_OK;
    if (!theta || !g || !v) return BOM_EINVAL;
    if (g_dtype != BOM_F32 && g_dtype != BOM_BF16) return BOM_EINVAL;
    if (!(beta2 >= 0.0f && beta2 < 1.0f) || !(eps >= 0.0f)) return BOM_EINVAL;
    if (!aligned16(theta) || !aligned16(g) || !aligned16(v) || (hvec && !aligned16(hvec)) ||
        (theta_bf16 && !aligned16(theta_bf16)))
        return BOM_ENOTSUP;
    const float inv_bc2 = inv_bias_correction(beta2, t);
    return static_cast<bom_status>(launch_update(theta, g, g_dtype == BOM_BF16, hvec, v, theta_bf16, n, lr, wd,
                                                 lambda, beta2, eps, inv_bc2, nullptr, 0.0f, nullptr,
                                                 static_cast<cudaStream_t>(stream)));
}

bom_status bom_sqnorm(bom_handle* h, const void* g, int32_t g_dtype, const float* hvec, float lambda, int64_t n,
                      double* sq, void* stream) {
    if (!h || n < 0 || !sq) return BOM_EINVAL;
    if (n == 0) return BOM_OK;
    if (!g || (g_dtype != BOM_F32 && g_dtype != BOM_BF16)) return BOM_EINVAL;
    if (!aligned16(g) || (hvec && !aligned16(hvec))) return BOM_ENOTSUP;
    return static_cast<bom_status>(launch_sqnorm(g, g_dtype == BOM_BF16, hvec, lambda, n, h->tel_part, sq,
                                                 static_cast<cudaStream_t>(stream)));
}

bom_status bom_update_clipped(float* theta, const void* g, int32_t g_dtype, const float* hvec, float* v,
                              uint16_t* theta_bf16, int64_t n, float lr, float wd, float lambda, float beta2,
                              float eps, int64_t t, const double* sq, float max_norm, void* stream) {
    if (n < 0 || t < 1 || !sq || !(max_norm > 0.0f)) return BOM_EINVAL;
    if (n == 0) return BOM_OK;
    if (!theta || !g || !v) return BOM_EINVAL;
    if (g_dtype != BOM_F32 && g_dtype != BOM_BF16) return BOM_EINVAL;
    if (!(beta2 >= 0.0f && beta2 < 1.0f) || !(eps >= 0.0f)) return BOM_EINVAL;
    if (!aligned16(theta) || !aligned16(g) || !aligned16(v) || (hvec && !aligned16(hvec)) ||
        (theta_bf16 && !aligned16(theta_bf16)))
        return BOM_ENOTSUP;
    const float inv_bc2 = inv_bias_correction(beta2, t);
    return static_cast<bom_status>(launch_update(theta, g, g_dtype == BOM_BF16, hvec, v, theta_bf16, n, lr, wd,
                                                 lambda, beta2, eps, inv_bc2, sq, max_norm, nullptr,
                                                 static_cast<cudaStream_t>(stream)));
}

bom_status bom_update_blockshared(float* theta, const void* g, int32_t g_dtype, const float* hvec, float* v_blocks,
                                  uint16_t* theta_bf16, int64_t n, int64_t block, float lr, float wd, float lambda,
                                  float beta2, float eps, int64_t t, void* stream) {
    if (n < 0 || t < 1 || block < 1) return BOM_EINVAL;
    if (n == 0) return BOM_OK;
    if (!theta || !g || !v_blocks) return BOM_EINVAL;
    if (g_dtype != BOM_F32 && g_dtype != BOM_BF16) return BOM_EINVAL;
    if (!(beta2 >= 0.0f && beta2 < 1.0f) || !(eps >= 0.0f)) return BOM_EINVAL;
    if (!aligned16(theta) || !aligned16(g) || (hvec && !aligned16(hvec)) || (theta_bf16 && !aligned16(theta_bf16)))
        return BOM_ENOTSUP;
    const float inv_bc2 = inv_bias_correction(beta2, t);
    return static_cast<bom_status>(launch_update_blockshared(theta, g, g_dtype == BOM_BF16, hvec, v_blocks, theta_bf16,
                                                             n, block, lr, wd, lambda, beta2, eps, inv_bc2,
                                                             static_cast<cudaStream_t>(stream)));
}

bom_status bom_gemm_bf16(const uint16_t* A, int64_t lda, int32_t a_mn_major, const uint16_t* B, int64_t ldb,
                         int32_t b_mn_major, float* D, int64_t ldd, int64_t M, int64_t N, int64_t K, float alpha,
                         void* stream) {
    if (!A || !B || !D || M < 1 || N < 1 || K < 0) return BOM_EINVAL;
    if ((ldd % 4) != 0 || !aligned16(D) || ldd < N) return BOM_ENOTSUP;
    GemmDesc g = gemm1(M, N, K, Operand{A, lda, a_mn_major != 0}, Operand{B, ldb, b_mn_major != 0});
    g.epi.alpha_const = alpha;
    g.epi.out = D;
    g.epi.ld_out = ldd;
    g.epi.out_f32 = 1;
    g.epi.sc = nullptr;
    return static_cast<bom_status>(launch_gemm_tc(g, static_cast<cudaStream_t>(stream)));
}

bom_status bom_trace(bom_handle* h, int32_t enable) {
    if (!h) return BOM_EINVAL;
    h->tracing = enable != 0;
    h->trace_n = 0;
    return BOM_OK;
}

int32_t bom_trace_read(bom_handle* h, bom_trace_entry* out, int32_t max, void* stream) {
    if (!h || (max > 0 && !out)) return -1;
    if (cudaStreamSynchronize(static_cast<cudaStream_t>(stream)) != cudaSuccess) return -1;
    for (int i = 0; i < h->trace_n && i < max; ++i) {
        const auto& r = h->trace[i];
        float ms = 0.0f;
        if (cudaEventElapsedTime(&ms, r.a, r.b) != cudaSuccess) return -1;
        out[i].name = r.name;
        out[i].flops = r.flops;
        out[i].bytes = r.bytes;
        out[i].ms = ms;
    }
    return h->trace_n;
}

int64_t bom_launch_count(void) { return static_cast<int64_t>(bom::g_launches.load()); }

const char* bom_status_string(bom_status s) {
    switch (s) {
        case BOM_OK: return "BOM_OK";
        case BOM_EINVAL: return "BOM_EINVAL: invalid argument";
        case BOM_ENOMEM: return "BOM_ENOMEM: device workspace allocation failed";
        case BOM_ECUDA: return "BOM_ECUDA: CUDA call failed";
        case BOM_ELABEL: return "BOM_ELABEL: label outside [0, d_out) that is not ignore_index";
        case BOM_EEMPTY: return "BOM_EEMPTY: no supervised outputs (N_t = 0)";
        case BOM_ETIMEOUT: return "BOM_ETIMEOUT: a bounded device wait ran out";
        case BOM_ENOTSUP: return "BOM_ENOTSUP: shape or alignment not supported";
        case BOM_ENONFINITE: return "BOM_ENONFINITE: non-finite logits (row log-sum-exp or label logit)";
        case BOM_ESHARD: return "BOM_ESHARD: another row shard of the sharded step latched an error";
    }
    return "unknown bom_status";
}

}  // extern "C"
