"""Pins of the oracle's global-norm clipping of the numerator (pretraining-
parameters appendix: clipping at 1.0; convergence appendix: the clipped
numerator feeds the adaptive update) against torch's own routines:
torch.nn.utils.clip_grad_norm_ for the factor, and clip_grad_norm_ followed by
torch.optim.AdamW(betas=(0, beta2)) for the clipped update at lambda = 0."""
import numpy as np
import torch

import oracle as O
from tests import _indep as X

B2, EPS = 0.999, 1e-8


def _tensors(rng, scale):
    return [rng.standard_normal(s) * scale for s in ((5, 7), (7,), (3, 5), (3,))]


def test_clip_factor_matches_torch_clip_grad_norm():
    rng = np.random.default_rng(0)
    for scale in (1e-3, 0.2, 1.0, 30.0):
        us = _tensors(rng, scale)
        ps = [torch.nn.Parameter(torch.zeros(u.shape, dtype=torch.float64)) for u in us]
        for p, u in zip(ps, us):
            p.grad = torch.tensor(u.copy())
        torch.nn.utils.clip_grad_norm_(ps, 1.0)
        c = O.clip_factor(us, 1.0)
        for p, u in zip(ps, us):
            assert X.rel_l2(c * u, p.grad.numpy()) < 1e-15
        norm = np.sqrt(sum((u ** 2).sum() for u in us))
        if norm <= 1.0:
            assert c == 1.0
        else:
            assert abs(np.sqrt(sum(((c * u) ** 2).sum() for u in us)) - 1.0) < 1e-5


def test_clipped_update_is_torch_clip_then_adamw_beta1_zero():
    rng = np.random.default_rng(1)
    thetas = _tensors(rng, 1.0)
    wds = [0.1, 0.0, 0.1, 0.0]
    ps = [torch.nn.Parameter(torch.tensor(t.copy())) for t in thetas]
    groups = [{"params": [p], "weight_decay": wd} for p, wd in zip(ps, wds)]
    opt = torch.optim.AdamW(groups, lr=1e-2, betas=(0.0, B2), eps=EPS)
    vs = [np.zeros(t.shape) for t in thetas]
    for t in range(1, 5):
        us = _tensors(rng, 0.5 * t)
        for p, u in zip(ps, us):
            p.grad = torch.tensor(u.copy())
        torch.nn.utils.clip_grad_norm_(ps, 1.0)
        opt.step()
        thetas, vs, c = O.bom_update_clipped(thetas, us, vs, 1e-2, wds, t, 1.0, B2, EPS)
        assert c < 1.0
        for th, p in zip(thetas, ps):
            assert X.rel_l2(th, p.detach().numpy()) < 1e-13
