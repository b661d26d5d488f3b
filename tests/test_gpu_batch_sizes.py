"""One handle, batches of different sizes.

The workspace of a handle is sized for max_rows, and a training loop feeds it
batches of any size up to that (the last batch of an epoch is short).  Each
step must read only its own rows: no per-row statistic, column partial or
cotangent left by a larger earlier batch may enter a smaller later one.  The
sequence below goes full -> about 2/7 -> 1 row -> 3/5 -> full on a handle
with spare rows, and every step is compared with the fp64 oracle on the
inputs that step read (its rows and the q left by the previous step).  A
batch above max_rows is refused on the host."""
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


@pytest.mark.parametrize("name", ["tiny_ragged_f32", "vision_small", "lm_head_small", "lm_mlp_small"])
def test_batch_size_changes_between_steps(name):
    wl = I.WORKLOADS[name]
    params = I.init_params(wl, seed=21)
    p64 = X.params_f64(wl, params)
    x, y = I.make_batch(wl, seed=21, step=1)
    y = y.copy()
    if y[0] == I.IGNORE_INDEX:
        y[0] = 1                        # the one-row batch must have a supervised row
    n_full = wl.n_rows
    gpu = G.GpuBom(wl, params, max_rows=n_full + 17)
    tol = G.TOL[wl.dtype]
    for t, n in enumerate([n_full, n_full * 2 // 7 + 1, 1, n_full * 3 // 5, n_full], start=1):
        q_prev = G.np64(gpu.q)
        gout = gpu.step(x[:n], y[:n], t)
        oref = G.oracle_step(wl, p64, x[:n], y[:n], q_prev, t)
        st = gout["stats"]
        assert st["code"] == B.BOM_OK, (t, n)
        assert st["n_t"] == oref["n_t"], (t, n)
        assert abs(st["loss"] - oref["ce"]) <= tol * abs(oref["ce"]) + 1e-6, (t, n)
        for key in ("s", "q", "qhat"):
            assert G.rel_l2(gout[key], oref[key]) < tol, (t, n, key)
        valid = oref["valid"]
        assert G.rel_l2(gout["lse"][valid], oref["lse"][valid]) < tol, (t, n)
        for k, (u, ref) in enumerate(zip(gout["grads"], oref["u"])):
            assert G.rel_l2(G.np64(u), ref) < tol, (t, n, k)


def test_batch_above_max_rows_is_refused():
    wl = I.TINY_RAGGED_F32
    params = I.init_params(wl, seed=22)
    x, y = I.make_batch(wl, seed=22, step=1)
    gpu = G.GpuBom(wl, params, max_rows=wl.n_rows - 5)
    q_before = gpu.q.clone()
    with pytest.raises(B.BomError) as e:
        gpu.step(x, y, 1)
    assert e.value.code == B.BOM_EINVAL
    torch.cuda.synchronize()
    assert torch.equal(gpu.q, q_before)
