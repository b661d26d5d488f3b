// Allocation-free column reduction.
//
// bom_colsum_noalloc runs the same two kernels that form the reprojection
// factors inside bom_step (colsum_{I_t}(H) and W^T qhat), but takes their
// scratch from a fixed device array instead of a workspace, so the call never
// allocates.  It serves callers that are not allowed to allocate device memory
// themselves: code running while a stream is captured into a CUDA graph in
// global capture mode (where cudaMalloc is an error), and runtimes that own all
// device memory through their own pool and forbid side allocations.
#include <mutex>

#include "kernels.h"

namespace bom {
namespace {

// Scratch of the partial column sums: row_blocks(n_rows) * n_cols floats at most.
constexpr int64_t kNoAllocScratchFloats = int64_t(1) << 20;  // 4 MiB
static __device__ __align__(256) float g_colsum_scratch[kNoAllocScratchFloats];
// Status block read by the kernels; it stays zero because nothing writes it.
static __device__ __align__(256) DevScalars g_noalloc_status;

constexpr int kMaxDevices = 64;
struct DeviceScratch {
    float* part = nullptr;
    DevScalars* sc = nullptr;
    bool ready = false;
};
DeviceScratch g_dev[kMaxDevices];
std::mutex g_mu;

// Device addresses of the two arrays for the current device, looked up once
// per device (host code cannot use the symbols' host-side names as pointers).
bom_status scratch_for_current_device(DeviceScratch** out) {
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return BOM_ECUDA;
    std::lock_guard<std::mutex> lock(g_mu);
    DeviceScratch& d = g_dev[dev];
    if (!d.ready) {
        void* p = nullptr;
        if (cudaGetSymbolAddress(&p, g_colsum_scratch) != cudaSuccess) return BOM_ECUDA;
        d.part = static_cast<float*>(p);
        if (cudaGetSymbolAddress(&p, g_noalloc_status) != cudaSuccess) return BOM_ECUDA;
        d.sc = static_cast<DevScalars*>(p);
        d.ready = true;
    }
    *out = &d;
    return BOM_OK;
}

}  // namespace
}  // namespace bom

extern "C" bom_status bom_colsum_noalloc(const void* x, int32_t dtype, int64_t ldx, int64_t n_rows, int64_t n_cols,
                                         const float* weights, float* out, void* stream) {
    using namespace bom;
    if (!x || !out || n_rows < 1 || n_cols < 1 || ldx < n_cols) return BOM_EINVAL;
    if (dtype != BOM_F32 && dtype != BOM_BF16) return BOM_EINVAL;
    if ((reinterpret_cast<uintptr_t>(x) & 15u) != 0) return BOM_ENOTSUP;
    // Each factor is bounded before the product is formed, so no size the
    // caller passes can overflow the check: the row ranges run along
    // gridDim.y (at most 65535) and each holds n_cols partial sums.
    if (n_cols > kNoAllocScratchFloats) return BOM_ENOTSUP;
    const int64_t ranges = n_rows / kRowBlock + (n_rows % kRowBlock != 0 ? 1 : 0);
    if (ranges > 65535 || ranges > kNoAllocScratchFloats / n_cols) return BOM_ENOTSUP;
    DeviceScratch* d = nullptr;
    const bom_status st = scratch_for_current_device(&d);
    if (st != BOM_OK) return st;
    // Every partial the second kernel reads is written by the first kernel of
    // the same call, so nothing left over from an earlier call is ever read.
    launch_colsum(x, dtype == BOM_F32 ? 1 : 0, ldx, n_rows, n_cols, nullptr, 0, weights, 1.0f, d->part, out, 1, d->sc,
                  static_cast<cudaStream_t>(stream));
    return cudaPeekAtLastError() == cudaSuccess ? BOM_OK : BOM_ECUDA;
}
