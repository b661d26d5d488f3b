"""bom_colsum_noalloc: the allocation-free column sum.

Some callers may not allocate device memory at the moment they need this
reduction: code running while its stream is captured into a CUDA graph in
global capture mode (where cudaMalloc is an error), and runtimes that hand out
every device byte from their own pool.  The entry point therefore works out of
a fixed scratch array inside the library.  Its result is checked here against
an fp64 numpy sum of the same input values (bf16 or fp32, times fp32 weights),
on two calls in a row that reuse the shared scratch, on the single-range path
(at most 128 rows, no finishing launch), at exactly its size limit, and inside
a global-mode stream capture after a first call outside it.

The file is named to run last, so a failure here cannot hide the results of
the other GPU tests in a run that stops at the first failure."""
import numpy as np
import pytest
import torch

from paper_2609_36738_gb300 import bom as B
from paper_2609_36738_gb300 import inputs as I
from tests import _gpu as G

pytestmark = pytest.mark.gpu

# fp32 accumulation over at most 65,536 rows of unit-scale values: relative
# error far below 1e-5 of the fp64 sum's norm
TOL = G.TOL["f32"]


@pytest.fixture(scope="module", autouse=True)
def _built():
    G.ensure_built()


def _case(seed, n, d, dtype, weighted):
    """Device input and weights, with the fp64 reference sum of the exact
    values the device sees."""
    rng = np.random.default_rng(seed)
    vals = rng.standard_normal((n, d), dtype=np.float32)
    if dtype == B.BOM_BF16:
        bits = I.bf16_bits(vals)
        x = G.to_dev(bits)
        x64 = I.bf16_to_f64(bits)
    else:
        x = G.to_dev(vals)
        x64 = vals.astype(np.float64)
    w = rng.standard_normal(n).astype(np.float32) if weighted else None
    ref = (w.astype(np.float64)[:, None] * x64).sum(axis=0) if weighted else x64.sum(axis=0)
    return x, (torch.from_numpy(w).to(G.DEV) if weighted else None), ref


def _run(x, dtype, n, d, w):
    out = torch.full((d,), float("nan"), dtype=torch.float32, device=G.DEV)
    B.bom_colsum_noalloc(x, dtype, d, n, d, w, out)
    return out


@pytest.mark.parametrize("dtype", [B.BOM_BF16, B.BOM_F32])
def test_noalloc_colsum_matches_fp64_sum_on_two_calls(dtype):
    # a multi-range call, then a different shape on the same scratch
    cases = [(1, 3001, 520, True), (2, 700, 2048, False)]
    outs = []
    for seed, n, d, weighted in cases:
        x, w, ref = _case(seed, n, d, dtype, weighted)
        outs.append((_run(x, dtype, n, d, w), ref))
    torch.cuda.synchronize()
    for out, ref in outs:
        assert torch.isfinite(out).all()
        assert G.rel_l2(G.np64(out), ref) < TOL


@pytest.mark.parametrize("dtype", [B.BOM_BF16, B.BOM_F32])
def test_noalloc_colsum_single_range(dtype):
    """At most 128 rows: one row range, whose blocks write the result directly."""
    for seed, n, d in ((3, 128, 264), (4, 1, 40), (5, 77, 1024)):
        x, w, ref = _case(seed, n, d, dtype, True)
        out = _run(x, dtype, n, d, w)
        torch.cuda.synchronize()
        assert G.rel_l2(G.np64(out), ref) < TOL


def test_noalloc_colsum_rejects_sizes_beyond_its_scratch():
    x = torch.zeros((16, 16), dtype=torch.bfloat16, device=G.DEV)
    out = torch.zeros(16, dtype=torch.float32, device=G.DEV)
    # ceil(n / 128) * n_cols above 2^20 floats: refused on the host
    with pytest.raises(B.BomError) as e:
        B.bom_colsum_noalloc(x, B.BOM_BF16, 4096, 128 * 600, 2048, None, out)
    assert e.value.code == B.BOM_ENOTSUP


def test_noalloc_colsum_at_the_scratch_limit():
    """ceil(n / 128) * n_cols = 2^20 exactly (65,536 rows x 2,048 columns) is
    accepted and matches the fp64 sum; one row more is refused."""
    n, d = 128 * 512, 2048
    x, _, _ = _case(6, n + 1, d, B.BOM_BF16, False)
    out = torch.full((d,), float("nan"), dtype=torch.float32, device=G.DEV)
    with pytest.raises(B.BomError) as e:
        B.bom_colsum_noalloc(x, B.BOM_BF16, d, n + 1, d, None, out)
    assert e.value.code == B.BOM_ENOTSUP
    B.bom_colsum_noalloc(x, B.BOM_BF16, d, n, d, None, out)
    torch.cuda.synchronize()
    ref = G.np64(x[:n]).sum(axis=0)
    assert torch.isfinite(out).all()
    assert G.rel_l2(G.np64(out), ref) < TOL


def test_noalloc_colsum_inside_a_global_mode_capture():
    """A first call outside any capture resolves the scratch address on this
    device; the same call then runs inside a stream capture in global mode
    (where an allocation would fail the capture) and the replayed graph gives
    the fp64 sum."""
    n, d = 2000, 768
    x, w, ref = _case(7, n, d, B.BOM_BF16, True)
    out = torch.full((d,), float("nan"), dtype=torch.float32, device=G.DEV)
    B.bom_colsum_noalloc(x, B.BOM_BF16, d, n, d, w, out)
    torch.cuda.synchronize()
    out.fill_(float("nan"))
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, capture_error_mode="global"):
        B.bom_colsum_noalloc(x, B.BOM_BF16, d, n, d, w, out)
    torch.cuda.synchronize()
    assert torch.isnan(out).all()   # capture executed nothing
    for _ in range(2):
        out.fill_(float("nan"))
        g.replay()
        torch.cuda.synchronize()
        assert G.rel_l2(G.np64(out), ref) < TOL
