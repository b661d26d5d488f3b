"""The oracle's sampled head-gradient helpers equal the rows of its full
reverse pass (they restate the same formulas on a subset of rows)."""
import numpy as np

import oracle as O
from paper_2609_36738_gb300 import inputs as I
from tests import _indep as X


def test_sampled_head_rows_match_full_backward():
    wl = I.LM_HEAD_SMALL
    params = X.params_f64(wl, I.init_params(wl, 4))
    xb, y = I.make_batch(wl, 4, 1)
    x = X.x_f64(wl, xb)
    q0 = np.random.default_rng(2).standard_normal(wl.vocab) * 0.01
    out = O.bom_step([], False, params, x, y, q0, 2)
    rows_v = np.array([0, 5, 77, wl.vocab - 1])
    rows_i = np.array([0, 3, 150, wl.n_rows - 1])
    gw = O.head_weight_grad_rows(out["R"], x, out["valid"], out["qhat"], out["n_t"], 0.5, rows_v)
    assert X.rel_l2(gw, out["u"][0][rows_v]) < 1e-13
    gi = O.head_input_grad_rows(out["R"], params[0], out["valid"], out["qhat"], out["n_t"], 0.5, rows_i)
    assert X.rel_l2(gi, out["dX_u"][rows_i]) < 1e-13
