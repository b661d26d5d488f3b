"""BOM-Adam-mini update kernel (bom_update_blockshared) against the oracle's
block-shared update (Section 3.5, composition with Adam-mini)."""
import numpy as np
import pytest
import torch

import oracle as O
from paper_2609_36738_gb300 import bom as B
from paper_2609_36738_gb300 import inputs as I
from tests import _gpu as G

pytestmark = pytest.mark.gpu

LAM, B2, EPS, LR, WD = 0.5, 0.999, 1e-8, 1e-3, 0.01
F = lambda x: float(np.float32(x))
LAMf, B2f, EPSf, LRf, WDf = F(LAM), F(B2), F(EPS), F(LR), F(WD)


@pytest.fixture(scope="module", autouse=True)
def _built():
    G.ensure_built()


def _close(th_gpu, theta0, ref_th, rel=1e-5):
    got = G.np64(th_gpu)
    ulp = np.spacing(np.abs(ref_th).astype(np.float32)).astype(np.float64)
    err = np.abs(got - ref_th)
    bound = 2 * ulp + rel * np.abs(ref_th - theta0)
    assert (err <= bound).all(), float((err / bound).max())


# (n, block): per-output-neuron rows of the vision head and LM shapes, a ragged
# last block, blocks that are not a multiple of 4, whole-tensor blocks and
# blocks of one element (elementwise BOM-AdamW).
# The register-resident kernel takes blocks of up to 8192 elements (d % 4 = 0).
# Larger blocks take the cluster kernel (eight CTAs per block) when there are
# at least as many blocks as cluster slots (201 blocks of 10_000; 171 odd-sized
# ones on its scalar path), else the grid-wide path: the 16-Mi-element
# whole-tensor block of a 4096 x 4096 weight, one aligned whole-tensor block,
# a few blocks with a ragged last one, and the odd-sized (50_001, 50_001).
# Small odd sizes take the scalar kernel.
CASES = [(3072 * 768, 768), (64 * 2048, 2048), (8 * 8192, 8192), (1000, 300), (29 * 7, 29), (50_001, 50_001),
         (4099, 1), (3, 5), (3 * 16384, 16384), (1 << 20, 1 << 20), (5 * 40_000 + 124, 40_000),
         (4096 * 4096, 4096 * 4096), (200 * 10_000 + 5_000, 10_000), (170 * 9_001 + 17, 9_001)]


@pytest.mark.parametrize("n,block", CASES)
@pytest.mark.parametrize("mode", ["g_and_h", "u_f32"])
def test_blockshared_update_matches_oracle(n, block, mode):
    theta, g, h, _ = I.update_sweep_host(n, seed=4)
    nb = -(-n // block)
    rng = np.random.default_rng(5)
    v0 = (rng.random(nb) * 1e-6).astype(np.float32)
    th = G.to_dev(theta)
    vb = G.to_dev(v0)
    sh = torch.empty(n, dtype=torch.bfloat16, device=G.DEV)
    t = 7
    if mode == "g_and_h":
        B.bom_update_blockshared(th, G.to_dev(g), B.BOM_BF16, G.to_dev(h), vb, sh, n, block, LR, WD, LAM, B2, EPS, t)
        u = O.mix_numerator(I.bf16_to_f64(g), h, LAMf)
    else:
        uf = (I.bf16_to_f64(g) + h).astype(np.float32)
        B.bom_update_blockshared(th, G.to_dev(uf), B.BOM_F32, None, vb, sh, n, block, LR, WD, LAM, B2, EPS, t)
        u = uf.astype(np.float64)
    torch.cuda.synchronize()
    ref_th, ref_v = O.bom_update_blockshared(theta, u, v0, block, LRf, WDf, t, B2f, EPSf)
    assert G.rel_l2(G.np64(vb), ref_v) < 1e-5
    _close(th, theta, ref_th)
    assert torch.equal(sh, th.to(torch.bfloat16))


def test_blockshared_trajectory_and_determinism():
    """Five steps on a [512, 768] weight with per-row blocks; a second run from
    the same state gives bit-identical theta and v."""
    rows, cols = 512, 768
    n = rows * cols
    theta, _, _, _ = I.update_sweep_host(n, seed=6)
    outs = []
    for rep in range(2):
        th = G.to_dev(theta)
        vb = torch.zeros(rows, dtype=torch.float32, device=G.DEV)
        ref_th, ref_v = theta.astype(np.float64), np.zeros(rows)
        for t in range(1, 6):
            _, g, h, _ = I.update_sweep_host(n, seed=100 + t)
            B.bom_update_blockshared(th, G.to_dev(g), B.BOM_BF16, G.to_dev(h), vb, None, n, cols, LR, WD, LAM, B2,
                                     EPS, t)
            ref_th, ref_v = O.bom_update_blockshared(ref_th, O.mix_numerator(I.bf16_to_f64(g), h, LAMf), ref_v, cols,
                                                     LRf, WDf, t, B2f, EPSf)
        torch.cuda.synchronize()
        assert G.rel_l2(G.np64(th), ref_th) < 1e-6
        assert G.rel_l2(G.np64(vb), ref_v) < 1e-5
        outs.append((th.clone(), vb.clone()))
    assert torch.equal(outs[0][0], outs[1][0]) and torch.equal(outs[0][1], outs[1][1])


@pytest.mark.parametrize("n,block", [(6 * 65_536 + 36, 65_536), (200 * 10_000 + 5_000, 10_000)])
def test_blockshared_large_blocks_are_deterministic(n, block):
    """Blocks spread over many CTAs (the grid-wide path for a few blocks, the
    cluster kernel for many) add their partial sums in a fixed order: two runs
    from the same state agree to the bit."""
    theta, g, h, _ = I.update_sweep_host(n, seed=8)
    outs = []
    for _ in range(2):
        th = G.to_dev(theta)
        vb = torch.zeros(-(-n // block), dtype=torch.float32, device=G.DEV)
        for t in range(1, 4):
            B.bom_update_blockshared(th, G.to_dev(g), B.BOM_BF16, G.to_dev(h), vb, None, n, block, LR, WD, LAM, B2,
                                     EPS, t)
        torch.cuda.synchronize()
        outs.append((th.clone(), vb.clone()))
    assert torch.equal(outs[0][0], outs[1][0]) and torch.equal(outs[0][1], outs[1][1])


def test_blockshared_rejects_bad_arguments():
    x = torch.zeros(8, device=G.DEV)
    with pytest.raises(B.BomError) as e:
        B.bom_update_blockshared(x, x, B.BOM_F32, None, x, None, 8, 0, LR, WD, LAM, B2, EPS, 1)
    assert e.value.code == B.BOM_EINVAL
    with pytest.raises(B.BomError) as e:
        B.bom_update_blockshared(x, x, B.BOM_F32, None, x, None, 8, 4, LR, WD, LAM, B2, EPS, 0)
    assert e.value.code == B.BOM_EINVAL
    with pytest.raises(B.BomError) as e:
        B.bom_update_blockshared(x.data_ptr() + 4, x, B.BOM_F32, None, x, None, 4, 4, LR, WD, LAM, B2, EPS, 1)
    assert e.value.code == B.BOM_ENOTSUP
    B.bom_update_blockshared(x, x, B.BOM_F32, None, x, None, 0, 4, LR, WD, LAM, B2, EPS, 1)   # n = 0: no-op
