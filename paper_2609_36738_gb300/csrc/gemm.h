// Host-side description of one GEMM of the BOM step and the two engines that
// run it: the tcgen05 tensor-core engine (bf16 operands) and the SIMT engine
// (fp32 operands, used by the fp32 configuration).
#pragma once
#include <cstdint>
#include <cuda_runtime.h>

#include "common.cuh"

namespace bom {

// A logical R x K operand.  K-major: element (r, k) at ptr[r*ld + k].
// MN-major: element (r, k) at ptr[k*ld + r].
struct Operand {
    const void* ptr;
    int64_t ld;
    bool mn_major;
};

// D[M, N] = sum over segments s of A_s[M, K_s] * B_s[N, K_s]^T, then the
// epilogue.  dual_b (EPI_SWIGLU_FWD only): each 256-column accumulator tile
// takes its first 128 B rows from B[0] and its last 128 from B[1], both at
// output column tile * 128, so one tile holds matching gate / up columns.
struct GemmDesc {
    int64_t M = 0, N = 0;
    int nseg = 1;
    Operand A[2] = {};
    Operand B[2] = {};
    int64_t K[2] = {0, 0};
    bool dual_b = false;
    int epi_kind = EPI_LINEAR;
    EpiParams epi = {};
    // Optional fp32 scratch for split-K (EPI_LINEAR only): when the output has
    // too few tiles to fill the GPU, the K range is split, fp32 partial tiles go
    // here and a fixed-order reduction applies the epilogue.
    float* splitk_ws = nullptr;
    int64_t splitk_ws_elems = 0;
};

// Returns BOM_OK or an error status (BOM_ENOTSUP for unsupported layouts,
// BOM_ECUDA for launch failures).
int launch_gemm_tc(const GemmDesc& g, cudaStream_t stream);
// One persistent launch over n <= 4 GEMMs with the same layout, epilogue
// kind and K and M > 128 (each GEMM launched alone otherwise).
int launch_gemm_tc_group(const GemmDesc* g, int n, cudaStream_t stream);
int launch_gemm_simt(const GemmDesc& g, cudaStream_t stream);
// One launch over n <= 4 GEMMs on the SIMT engine.
int launch_gemm_simt_group(const GemmDesc* g, int n, cudaStream_t stream);

// Number of column tiles of EPI_LOGITS statistics produced per row.
int64_t tc_logit_tiles(int64_t N);

int device_sm_count();

}  // namespace bom
