"""The tcgen05 GEMM engine (bom_gemm_bf16) against an fp64 matmul of the same
bf16 operands, for every operand layout, on shapes spanning several tiles
(narrow 128 x 64 and CTA-pair 256 x 256) with ragged tails, K tails and the
empty-K case."""
import numpy as np
import pytest
import torch

from paper_2609_36738_gb300 import bom as B
from paper_2609_36738_gb300 import inputs as I
from tests import _gpu as G

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    G.ensure_built()


def _rup(a, b):
    return (a + b - 1) // b * b


def _operand(rng, rows, K, mn_major):
    """Logical rows x K bf16 operand stored K-major [rows, ldk] or MN-major [K, ldm]."""
    logical = rng.standard_normal((rows, K), dtype=np.float32)
    bits = I.bf16_bits(logical)
    val = I.bf16_to_f64(bits)
    if mn_major:
        ld = _rup(rows, 8)
        store = np.zeros((max(K, 1), ld), dtype=np.uint16)
        store[:K, :rows] = bits.T
    else:
        ld = _rup(max(K, 1), 8)
        store = np.zeros((rows, ld), dtype=np.uint16)
        store[:, :K] = bits
    return G.to_dev(store), ld, val


@pytest.mark.parametrize("a_mn,b_mn", [(0, 0), (0, 1), (1, 0), (1, 1)])
# The first five shapes have few enough 256 x 256 tiles to run on 128 x 64
# single-CTA tiles when A is K-major; the last two have enough to keep the
# CTA-pair tiles, with ragged M, N and K (130 rows: a pair whose odd CTA has
# two valid rows).
@pytest.mark.parametrize("M,N,K", [(128, 256, 64), (300, 520, 200), (1, 7, 8), (257, 1000, 136), (640, 768, 1024),
                                   (1000, 2500, 300), (130, 9000, 96)])
def test_gemm_layouts(a_mn, b_mn, M, N, K):
    rng = np.random.default_rng(M * 7 + N * 13 + K)
    A, lda, Av = _operand(rng, M, K, a_mn)
    Bt, ldb, Bv = _operand(rng, N, K, b_mn)
    ldd = _rup(N, 4)
    D = torch.full((M, ldd), float("nan"), dtype=torch.float32, device=G.DEV)
    B.bom_gemm_bf16(A, lda, a_mn, Bt, ldb, b_mn, D, ldd, M, N, K, 0.5)
    torch.cuda.synchronize()
    ref = 0.5 * Av @ Bv.T
    got = G.np64(D)[:, :N]
    assert np.isfinite(got).all()
    assert G.rel_l2(got, ref) < 1e-5
    # columns beyond N are never written
    if ldd > N:
        assert torch.isnan(D[:, N:]).all()


def test_gemm_empty_k_writes_zeros():
    A = torch.zeros((16, 8), dtype=torch.bfloat16, device=G.DEV)
    D = torch.full((16, 32), 7.0, dtype=torch.float32, device=G.DEV)
    B.bom_gemm_bf16(A, 8, 0, A, 8, 0, D, 32, 16, 16, 0, 1.0)
    torch.cuda.synchronize()
    assert (D[:, :16] == 0).all() and (D[:, 16:] == 7).all()


def test_gemm_rejects_unaligned_pitch():
    A = torch.zeros((16, 12), dtype=torch.bfloat16, device=G.DEV)
    D = torch.zeros((16, 16), dtype=torch.float32, device=G.DEV)
    with pytest.raises(B.BomError) as e:
        B.bom_gemm_bf16(A, 12, 0, A, 12, 0, D, 16, 16, 16, 12, 1.0)
    assert e.value.code == B.BOM_ENOTSUP
