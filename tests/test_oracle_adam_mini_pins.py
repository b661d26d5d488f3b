"""Pins of the oracle's BOM-Adam-mini update (Section 3.5, composition with
Adam-mini; optimizer-implementation appendix) against facts that do not come
from the oracle itself:

* blocks of one element are elementwise BOM-AdamW, i.e. torch.optim.AdamW
  with beta1 = 0 fed u as the gradient (library special case);
* a block whose |u| is constant shares v with nothing else in effect, so it
  matches the elementwise update (checks the block boundaries, ragged last
  block included);
* at t = 1 with eps = 0 and no decay, every block's step has root-mean-square
  exactly eta, and rescaling u within a block leaves its steps unchanged."""
import numpy as np
import pytest
import torch

import oracle as O
from tests import _indep as X

B2, EPS = 0.999, 1e-8


def test_block_of_one_is_torch_adamw_with_beta1_zero():
    rng = np.random.default_rng(0)
    n, lr, wd = 37, 1e-2, 0.1
    theta = rng.standard_normal(n)
    p = torch.nn.Parameter(torch.tensor(theta.copy()))
    opt = torch.optim.AdamW([p], lr=lr, betas=(0.0, B2), eps=EPS, weight_decay=wd)
    v = np.zeros(n)
    for t in range(1, 4):
        u = rng.standard_normal(n) * 10.0 ** rng.uniform(-3, 0, n)
        p.grad = torch.tensor(u)
        opt.step()
        theta, v = O.bom_update_blockshared(theta, u, v, 1, lr, wd, t, B2, EPS)
        assert X.rel_l2(theta, p.detach().numpy()) < 1e-14


@pytest.mark.parametrize("n,block", [(60, 12), (61, 12), (50, 50), (7, 3)])
def test_constant_magnitude_blocks_match_elementwise(n, block):
    rng = np.random.default_rng(1)
    nb = -(-n // block)
    theta = rng.standard_normal(n)
    v_el, v_bl = np.zeros(n), np.zeros(nb)
    th_el, th_bl = theta.copy(), theta.copy()
    for t in range(1, 5):
        mag = np.repeat(10.0 ** rng.uniform(-3, 1, nb), block)[:n]
        u = mag * np.where(rng.random(n) < 0.5, -1.0, 1.0)
        th_el, v_el = O.bom_update(th_el, u, v_el, 1e-3, 0.01, t, B2, EPS)
        th_bl, v_bl = O.bom_update_blockshared(th_bl, u, v_bl, block, 1e-3, 0.01, t, B2, EPS)
        assert X.rel_l2(th_bl, th_el) < 1e-15
        assert X.rel_l2(np.repeat(v_bl, block)[:n], v_el) < 1e-15


def test_first_step_block_rms_is_lr_and_scale_free():
    rng = np.random.default_rng(2)
    n, block, lr = 40, 8, 3e-3
    theta = rng.standard_normal(n)
    u = rng.standard_normal(n)
    new, _ = O.bom_update_blockshared(theta, u, np.zeros(n // block), block, lr, 0.0, 1, B2, 0.0)
    d = (new - theta).reshape(-1, block)
    assert np.allclose(np.sqrt((d ** 2).mean(axis=1)), lr, rtol=1e-14, atol=0)
    scale = np.repeat(10.0 ** rng.uniform(-4, 4, n // block), block)
    th_a, th_b, v_a, v_b = theta.copy(), theta.copy(), np.zeros(n // block), np.zeros(n // block)
    for t in range(1, 4):
        w = rng.standard_normal(n)
        th_a, v_a = O.bom_update_blockshared(th_a, w, v_a, block, lr, 0.0, t, B2, 0.0)
        th_b, v_b = O.bom_update_blockshared(th_b, w * scale, v_b, block, lr, 0.0, t, B2, 0.0)
        assert X.rel_l2(th_b, th_a) < 1e-14


def test_state_is_one_entry_per_block_and_errors():
    with pytest.raises(O.OracleError):
        O.bom_update_blockshared(np.zeros(10), np.zeros(10), np.zeros(3), 4, 1e-3, 0.0, 0)
    with pytest.raises(O.OracleError):
        O.bom_update_blockshared(np.zeros(10), np.zeros(10), np.zeros(2), 4, 1e-3, 0.0, 1)
    with pytest.raises(O.OracleError):
        O.bom_update_blockshared(np.zeros(10), np.zeros(10), np.zeros(10), 0, 1e-3, 0.0, 1)
