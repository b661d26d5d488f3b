"""Global-norm clipping on the GPU (bom_sqnorm + bom_update_clipped) against the
oracle's clipped update (pretraining-parameters appendix: clipping at 1.0;
convergence appendix: the clipped numerator feeds the update)."""
import numpy as np
import pytest
import torch

import oracle as O
from paper_2609_36738_gb300 import bom as B
from paper_2609_36738_gb300 import inputs as I
from tests import _gpu as G

pytestmark = pytest.mark.gpu
LAM, B2, EPS, LR = 0.5, 0.999, 1e-8, 1e-3
F = lambda x: float(np.float32(x))


@pytest.fixture(scope="module", autouse=True)
def _built():
    G.ensure_built()


def _handle():
    return B.BomModel(B.config_for(I.TINY_MLP_F32))


@pytest.mark.parametrize("scale,max_norm", [(1e-3, 1.0), (1.0, 1.0), (50.0, 0.5)])
def test_clipped_update_over_three_ranges(scale, max_norm):
    """Three tensors (sizes 1_000_003, 4096, 7) clipped together; u = (1-lambda) g + lambda h."""
    m = _handle()
    sizes = [1_000_003, 4096, 7]
    wds = [0.1, 0.0, 0.1]
    data = []
    for k, n in enumerate(sizes):
        theta, g, h, v = I.update_sweep_host(n, seed=20 + k)
        h = (h * scale).astype(np.float32)
        g = I.bf16_bits((I.bf16_to_f32(g) * scale).astype(np.float32))
        data.append((theta, g, h, v))
    sq = torch.zeros(1, dtype=torch.float64, device=G.DEV)
    dev = []
    for theta, g, h, v in data:
        gd, hd = G.to_dev(g), G.to_dev(h)
        B.bom_sqnorm(m.h, gd, B.BOM_BF16, hd, LAM, theta.size, sq)
        dev.append((G.to_dev(theta), gd, hd, G.to_dev(v)))
    t = 3
    for (th, gd, hd, vd), wd in zip(dev, wds):
        B.bom_update_clipped(th, gd, B.BOM_BF16, hd, vd, None, th.numel(), LR, wd, LAM, B2, EPS, t, sq, max_norm)
    torch.cuda.synchronize()
    us = [O.mix_numerator(I.bf16_to_f64(g), h, F(LAM)) for _, g, h, _ in data]
    sq_ref = sum(float((u ** 2).sum()) for u in us)
    assert abs(G.np64(sq)[0] - sq_ref) <= 1e-5 * sq_ref
    ths, vs, c = O.bom_update_clipped([d[0] for d in data], us, [d[3] for d in data], F(LR), [F(w) for w in wds],
                                      t, F(max_norm), F(B2), F(EPS))
    assert (c < 1.0) == (np.sqrt(sq_ref) > max_norm)
    for (th, _, _, vd), (theta0, _, _, _), ref_th, ref_v in zip(dev, data, ths, vs):
        got = G.np64(th)
        ulp = np.spacing(np.abs(ref_th).astype(np.float32)).astype(np.float64)
        assert np.all(np.abs(got - ref_th) <= 2 * ulp + 1e-5 * np.abs(ref_th - theta0))
        assert G.rel_l2(G.np64(vd), ref_v) < 1e-5


def test_clip_inactive_is_bitwise_bom_update():
    """Norm below max_norm: the clipped update is the plain update, bit for bit."""
    m = _handle()
    n = 100_001
    theta, g, h, v = I.update_sweep_host(n, seed=30)
    sq = torch.zeros(1, dtype=torch.float64, device=G.DEV)
    gd, hd = G.to_dev(g), G.to_dev(h)
    B.bom_sqnorm(m.h, gd, B.BOM_BF16, hd, LAM, n, sq)
    a_th, a_v = G.to_dev(theta), G.to_dev(v)
    b_th, b_v = G.to_dev(theta), G.to_dev(v)
    B.bom_update_clipped(a_th, gd, B.BOM_BF16, hd, a_v, None, n, LR, 0.01, LAM, B2, EPS, 2, sq, 1e6)
    B.bom_update(b_th, gd, B.BOM_BF16, hd, b_v, None, n, LR, 0.01, LAM, B2, EPS, 2)
    torch.cuda.synchronize()
    assert torch.equal(a_th, b_th) and torch.equal(a_v, b_v)


def test_clip_argument_checks():
    m = _handle()
    x = torch.zeros(8, device=G.DEV)
    sq = torch.zeros(1, dtype=torch.float64, device=G.DEV)
    with pytest.raises(B.BomError) as e:
        B.bom_update_clipped(x, x, B.BOM_F32, None, x, None, 8, LR, 0.0, LAM, B2, EPS, 1, sq, 0.0)
    assert e.value.code == B.BOM_EINVAL
    with pytest.raises(B.BomError) as e:
        B.bom_update_clipped(x, x, B.BOM_F32, None, x, None, 8, LR, 0.0, LAM, B2, EPS, 1, None, 1.0)
    assert e.value.code == B.BOM_EINVAL
    with pytest.raises(B.BomError) as e:
        B.bom_sqnorm(m.h, x.data_ptr() + 4, B.BOM_F32, None, LAM, 4, sq)
    assert e.value.code == B.BOM_ENOTSUP
