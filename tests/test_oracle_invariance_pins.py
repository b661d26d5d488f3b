"""Batch invariances of the oracle's step that the paper's definitions fix.

s_t, q_t and the surrogate L_mix are means over the supervised set I_t
(Algorithm 1; Section 3.2; the LM construction appendix), so

- permuting the rows of a batch (labels with them) changes none of s_t, q_t,
  qhat_t, the CE loss, N_t or u, and permutes the per-row log-sum-exp;
- duplicating a batch (every row twice, ignored rows included) doubles N_t
  and changes no mean: s_t, q_t, CE and u stay the same.

A plausible mistake breaks one of them: a label paired with the wrong row
breaks the permutation invariance, a sum where the paper has a mean breaks
the duplication invariance.  (A count of all rows instead of N_t scales both
sides alike; the batch-decomposition and autograd pins catch that one.)  A
mutation test below plants each of the two mistakes in a restatement of s_t
and checks that an invariance, not a known answer, rejects it.
"""
import numpy as np
import pytest

import oracle as O
from paper_2609_36738_gb300 import inputs as I
from tests import _indep as X


def _step(wl, params, x, y, q_prev, t=4):
    return O.bom_step(X.oracle_layers(wl), wl.head_bias, params, x, y, q_prev, t)


def _inputs(wl, seed):
    params = X.params_f64(wl, I.init_params(wl, seed))
    xb, y = I.make_batch(wl, seed, 2)
    x = X.x_f64(wl, xb)
    y = y.copy()
    y[::7] = I.IGNORE_INDEX   # N_t < n on every workload
    rng = np.random.default_rng(seed + 5)
    q_prev = 0.03 * rng.standard_normal(wl.vocab)
    q_prev -= q_prev.mean()
    return params, x, y, q_prev


def _close(a, b, tol=1e-12):
    a, b = np.asarray(a, np.float64), np.asarray(b, np.float64)
    return np.linalg.norm(a - b) <= tol * max(np.linalg.norm(b), 1e-300)


@pytest.mark.parametrize("name", ["tiny_ragged_f32", "tiny_norm_f32", "vision_small", "lm_mlp_small"])
def test_row_permutation_changes_nothing_but_row_order(name):
    wl = I.WORKLOADS[name]
    params, x, y, q_prev = _inputs(wl, 31)
    perm = np.random.default_rng(32).permutation(x.shape[0])
    a = _step(wl, params, x, y, q_prev)
    b = _step(wl, params, x[perm], y[perm], q_prev)
    assert a["n_t"] == b["n_t"]
    for key in ("s", "q", "qhat"):
        assert _close(a[key], b[key]), key
    assert abs(a["ce"] - b["ce"]) <= 1e-12 * abs(a["ce"])
    assert _close(a["lse"][perm], b["lse"])
    for ua, ub in zip(a["u"], b["u"]):
        assert _close(ua, ub)


@pytest.mark.parametrize("name", ["tiny_ragged_f32", "tiny_norm_f32", "vision_small", "lm_mlp_small"])
def test_duplicated_batch_keeps_every_mean(name):
    wl = I.WORKLOADS[name]
    params, x, y, q_prev = _inputs(wl, 33)
    a = _step(wl, params, x, y, q_prev)
    b = _step(wl, params, np.concatenate([x, x]), np.concatenate([y, y]), q_prev)
    assert b["n_t"] == 2 * a["n_t"]
    assert a["n_t"] < x.shape[0]
    for key in ("s", "q", "qhat"):
        assert _close(a[key], b[key]), key
    assert abs(a["ce"] - b["ce"]) <= 1e-12 * abs(a["ce"])
    for ua, ub in zip(a["u"], b["u"]):
        assert _close(ua, ub)


def test_invariances_catch_planted_mistakes():
    """Plant a mistake in a restatement of s_t (the oracle itself is left
    alone) and check that the invariances above reject it."""
    wl = I.TINY_RAGGED_F32
    params, x, y, q_prev = _inputs(wl, 34)
    layers = X.oracle_layers(wl)
    Z = O.forward(layers, wl.head_bias, params, x)[0]

    def s_of(Zm, ym, mistake):
        valid, n_t = O.supervised_set(ym, wl.vocab)
        R = O.residuals(Zm, ym, valid)
        if mistake == "sum":
            return R.sum(axis=0)
        if mistake == "shifted_label":
            R = O.residuals(Zm, np.roll(ym, 1), O.supervised_set(np.roll(ym, 1), wl.vocab)[0])
            return R[:-1].sum(axis=0) / n_t
        return O.batch_mean_residual(R, n_t)

    perm = np.random.default_rng(35).permutation(x.shape[0])
    Zd, yd = np.concatenate([Z, Z]), np.concatenate([y, y])
    ok = s_of(Z, y, None)
    assert _close(ok, s_of(Z[perm], y[perm], None)) and _close(ok, s_of(Zd, yd, None))
    # a sum instead of the mean: caught by duplication
    assert not _close(s_of(Z, y, "sum"), s_of(Zd, yd, "sum"))
    # labels paired with the neighbouring row: caught by permutation
    assert not _close(s_of(Z, y, "shifted_label"), s_of(Z[perm], y[perm], "shifted_label"))
