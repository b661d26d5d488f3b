"""BOM-AdamW update kernel (bom_update) against the oracle's update
(Section 3.4; Algorithm 1, last two steps)."""
import numpy as np
import pytest
import torch

import oracle as O
from paper_2609_36738_gb300 import bom as B
from paper_2609_36738_gb300 import inputs as I
from tests import _gpu as G

pytestmark = pytest.mark.gpu

LAM, B2, EPS, LR, WD, T = 0.5, 0.999, 1e-8, 1e-3, 0.01, 10
# The C ABI takes the coefficients as fp32: the oracle gets those same values.
F = lambda x: float(np.float32(x))
LAMf, B2f, EPSf, LRf, WDf = F(LAM), F(B2), F(EPS), F(LR), F(WD)


def _assert_step_close(th_gpu, theta0, ref_th, rel=1e-5):
    """Updated fp32 theta within one ulp of the fp64 result plus a relative
    error of the step itself (the ulp of theta bounds how exactly an fp32
    parameter can take a small step)."""
    got = G.np64(th_gpu)
    ulp = np.spacing(np.abs(ref_th).astype(np.float32)).astype(np.float64)
    err = np.abs(got - ref_th)
    bound = ulp + rel * np.abs(ref_th - theta0)
    assert (err <= bound).all(), float((err / bound).max())


@pytest.fixture(scope="module", autouse=True)
def _built():
    G.ensure_built()


def _run(theta, g_bits_or_f32, h, v, shadow=False, t=T, lr=LR, wd=WD):
    th = G.to_dev(theta)
    gd = G.to_dev(g_bits_or_f32)
    hd = G.to_dev(h) if h is not None else None
    vd = G.to_dev(v)
    sh = torch.empty(theta.shape, dtype=torch.bfloat16, device=G.DEV) if shadow else None
    gt = B.BOM_BF16 if g_bits_or_f32.dtype == np.uint16 else B.BOM_F32
    B.bom_update(th, gd, gt, hd, vd, sh, theta.size, lr, wd, LAM, B2, EPS, t)
    torch.cuda.synchronize()
    return th, vd, sh


@pytest.mark.parametrize("n", [1, 3, 4, 1001, 10_000_000])
def test_update_g_and_h(n):
    theta, g, h, v = I.update_sweep_host(n, seed=1)
    th, vd, sh = _run(theta, g, h, v, shadow=True)
    ref_th, ref_v = O.bom_update_gh(theta, I.bf16_to_f64(g), h, v, LRf, WDf, LAMf, T, B2f, EPSf)
    assert G.rel_l2(G.np64(th), ref_th) < 1e-6
    assert G.rel_l2(G.np64(vd), ref_v) < 1e-6
    _assert_step_close(th, theta, ref_th)
    # bf16 copy is the rounded updated theta
    assert torch.equal(sh, th.to(torch.bfloat16))


def test_update_numerator_given_f32_first_step():
    """t = 1 with v = 0 and omega = 0: delta = -lr u / (|u| + eps)."""
    rng = np.random.default_rng(3)
    n = 4099
    theta = rng.standard_normal(n).astype(np.float32)
    u = (rng.standard_normal(n) * 1e-3).astype(np.float32)
    v = np.zeros(n, np.float32)
    th, vd, _ = _run(theta, u, None, v, t=1, wd=0.0)
    ref_th, ref_v = O.bom_update(theta, u, v, LRf, 0.0, 1, B2f, EPSf)
    _assert_step_close(th, theta, ref_th)
    assert G.rel_l2(G.np64(vd), ref_v) < 1e-6


def test_update_zero_length_is_noop():
    x = torch.zeros(4, device=G.DEV)
    B.bom_update(x, x, B.BOM_F32, None, x, None, 0, LR, WD, LAM, B2, EPS, 1)


def test_update_rejects_bad_arguments():
    x = torch.zeros(8, device=G.DEV)
    with pytest.raises(B.BomError):
        B.bom_update(x, x, B.BOM_F32, None, x, None, 8, LR, WD, LAM, B2, EPS, 0)   # t < 1
    with pytest.raises(B.BomError):
        B.bom_update(x[1:], x, B.BOM_F32, None, x, None, 4, LR, WD, LAM, B2, EPS, 1)  # unaligned


@pytest.mark.slow
def test_update_full_size_sampled():
    """1e9 elements (the largest sweep size): inputs drawn on the device, outputs
    checked against the oracle at 4096 sampled indices plus the ragged tail."""
    n = I.UPDATE_SIZES[-1] + 3
    theta, g, h, v = I.update_sweep_device(n, seed=2, device=G.DEV)
    rng = np.random.default_rng(4)
    idx = np.concatenate([rng.integers(0, n, 4096), np.arange(n - 7, n)])
    it = torch.from_numpy(idx).to(G.DEV)
    before = [G.np64(a[it]) for a in (theta, g, h, v)]
    B.bom_update(theta, g, B.BOM_BF16, h, v, None, n, LR, WD, LAM, B2, EPS, T)
    torch.cuda.synchronize()
    ref_th, ref_v = O.bom_update_gh(before[0], before[1], before[2], before[3], LRf, WDf, LAMf, T, B2f, EPSf)
    _assert_step_close(theta[it], before[0], ref_th)
    assert G.rel_l2(G.np64(v[it]), ref_v) < 1e-6
