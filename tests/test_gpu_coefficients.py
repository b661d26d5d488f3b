"""bom_step at the degenerate settings of the method's coefficients, against
the fp64 oracle on the same seeded inputs.

- lambda = 0: the cotangent is the plain CE residual, so u = g (Eq.
  mix-gradient with no momentum term);
- lambda = 1: only the momentum term is left, u = h = Jbar^T qhat;
- beta1 = 0: the task-space EMA keeps no history, q_t = qhat_t = s_t
  (Section 3.2); on the GPU this holds bit for bit, since q = 0 * q + 1 * s
  and the bias correction 1/(1 - 0^t) is exactly 1;
- an interior pair (0.3, 0.95) whose fp32 values are not short binary
  fractions.

The coefficients cross the ABI as fp32; the oracle gets the same fp32-rounded
values.  Tolerances are those of the single-step parity tests."""
import numpy as np
import pytest
import torch

from paper_2609_36738_gb300 import bom as B
from paper_2609_36738_gb300 import inputs as I
from tests import _gpu as G
from tests import _indep as X

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    G.ensure_built()


def _f32(v):
    return float(np.float32(v))


@pytest.mark.parametrize("name", ["tiny_ragged_f32", "lm_head_small", "lm_mlp_small"])
@pytest.mark.parametrize("lam,beta1", [(0.0, 0.9), (1.0, 0.9), (0.5, 0.0), (0.3, 0.95)])
@pytest.mark.parametrize("mode", [B.BOM_OUT_U, B.BOM_OUT_G_AND_H])
def test_step_at_coefficient_extremes(name, lam, beta1, mode):
    wl = I.WORKLOADS[name]
    lam, beta1 = _f32(lam), _f32(beta1)
    params = I.init_params(wl, seed=11)
    p64 = X.params_f64(wl, params)
    x, y = I.make_batch(wl, seed=11, step=1)
    rng = np.random.default_rng(12)
    q0 = (rng.standard_normal(wl.vocab) * 0.01).astype(np.float32)
    q0 -= q0.mean(dtype=np.float64).astype(np.float32)
    gpu = G.GpuBom(wl, params, out_mode=mode, lam=lam, beta1=beta1)
    gpu.q.copy_(torch.from_numpy(q0))
    t = 3
    gout = gpu.step(x, y, t)
    oref = G.oracle_step(wl, p64, x, y, q0.astype(np.float64), t, lam=lam, beta1=beta1)
    tol = G.TOL[wl.dtype]

    st = gout["stats"]
    assert st["code"] == B.BOM_OK
    assert st["n_t"] == oref["n_t"]
    assert abs(st["loss"] - oref["ce"]) <= tol * abs(oref["ce"]) + 1e-6
    for key in ("s", "q", "qhat"):
        assert G.rel_l2(gout[key], oref[key]) < tol, key
    if beta1 == 0.0:
        assert np.array_equal(gout["q"], gout["s"]) and np.array_equal(gout["qhat"], gout["s"])
    if mode == B.BOM_OUT_G_AND_H:
        for k, (g, ref) in enumerate(zip(gout["grads"], oref["g"])):
            assert G.rel_l2(G.np64(g), ref) < tol, f"g[{k}]"
        for k, (h, ref) in enumerate(zip(gout["h"], oref["h"])):
            assert G.rel_l2(G.np64(h), ref) < tol, f"h[{k}]"
    else:
        want = oref["g"] if lam == 0.0 else oref["h"] if lam == 1.0 else oref["u"]
        for k, (u, ref) in enumerate(zip(gout["grads"], want)):
            assert G.rel_l2(G.np64(u), ref) < tol, f"u[{k}]"
