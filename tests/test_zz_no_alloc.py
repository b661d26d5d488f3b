"""bom_colsum_noalloc: the allocation-free column sum, for callers that may not
allocate device memory (stream capture in global mode, externally managed
device memory).  Its result must match the library's GEMM entry point
bom_gemm_bf16 computing the same weighted sum as a 1-row GEMM, on two calls in
a row that reuse the library's fixed scratch array.

The file is named to run last, so a failure here cannot hide the results of
the other GPU tests in a run that stops at the first failure."""
import numpy as np
import pytest
import torch

from paper_2609_36738_gb300 import bom as B
from paper_2609_36738_gb300 import inputs as I
from tests import _gpu as G

pytestmark = pytest.mark.gpu

TOL = G.TOL["f32"]   # both sides sum exact bf16 x bf16 products in fp32


@pytest.fixture(scope="module", autouse=True)
def _built():
    G.ensure_built()


def _rup(a, b):
    return (a + b - 1) // b * b


def _case(seed, n, d, weighted):
    rng = np.random.default_rng(seed)
    x_bits = I.bf16_bits(rng.standard_normal((n, d), dtype=np.float32))
    x = G.to_dev(x_bits)
    if weighted:
        # weights exactly representable in bf16, so the GEMM operand is exact too
        w_bits = I.bf16_bits(rng.standard_normal(n, dtype=np.float32))
    else:
        w_bits = I.bf16_bits(np.ones(n, dtype=np.float32))
    w32 = torch.from_numpy(I.bf16_to_f32(w_bits)).to(G.DEV)
    # reference through the existing entry point: D[1, d] = w^T X as a GEMM with
    # A = w (1 x n, K-major) and B = X (d x n, stored MN-major as X itself)
    lda = _rup(n, 8)
    a = np.zeros((1, lda), dtype=np.uint16)
    a[0, :n] = w_bits
    ref = torch.full((1, _rup(d, 4)), float("nan"), dtype=torch.float32, device=G.DEV)
    B.bom_gemm_bf16(G.to_dev(a), lda, 0, x, d, 1, ref, ref.shape[1], 1, d, n, 1.0)
    return x, (w32 if weighted else None), ref[0, :d]


def test_noalloc_colsum_matches_gemm_entry_on_two_calls():
    cases = [(1, 3001, 520, True), (2, 700, 2048, False)]
    for seed, n, d, weighted in cases:
        x, w, ref = _case(seed, n, d, weighted)
        out = torch.full((d,), float("nan"), dtype=torch.float32, device=G.DEV)
        B.bom_colsum_noalloc(x, B.BOM_BF16, d, n, d, w, out)
        torch.cuda.synchronize()
        assert torch.isfinite(out).all()
        assert G.rel_l2(G.np64(out), G.np64(ref)) < TOL


def test_noalloc_colsum_rejects_sizes_beyond_its_scratch():
    x = torch.zeros((16, 16), dtype=torch.bfloat16, device=G.DEV)
    out = torch.zeros(16, dtype=torch.float32, device=G.DEV)
    # ceil(n / 128) * n_cols above 2^20 floats: refused on the host
    with pytest.raises(B.BomError) as e:
        B.bom_colsum_noalloc(x, B.BOM_BF16, 4096, 128 * 600, 2048, None, out)
    assert e.value.code == B.BOM_ENOTSUP


def test_noalloc_colsum_at_the_scratch_limit():
    """ceil(n / 128) * n_cols = 2^20 exactly (65,536 rows x 2,048 columns) is
    accepted and matches the GEMM entry; one row more is refused."""
    n, d = 128 * 512, 2048
    x, _, ref = _case(3, n + 1, d, False)
    out = torch.full((d,), float("nan"), dtype=torch.float32, device=G.DEV)
    with pytest.raises(B.BomError) as e:
        B.bom_colsum_noalloc(x, B.BOM_BF16, d, n + 1, d, None, out)
    assert e.value.code == B.BOM_ENOTSUP
    # the first n rows: the reference is the full sum minus the last row
    B.bom_colsum_noalloc(x, B.BOM_BF16, d, n, d, None, out)
    torch.cuda.synchronize()
    want = G.np64(ref) - G.np64(x[n].float())
    assert torch.isfinite(out).all()
    assert G.rel_l2(G.np64(out), want) < TOL
