"""Pins of the oracle's drift telemetry and own-step control (Section 3.3,
Eq. drift-telemetry; stale-control and drift-measurement appendices) against
facts the paper or mathematics fix:

* Jbar^T s from finite-difference Jacobians of an independent torch forward;
* at t = 1, Mhat_1 = Jbar_1^T s_1 = h_1 for any model (qhat_1 = s_1);
* on the classifier bias Jbar_b = I, so Mhat_t = qhat_t on any trajectory;
* a linear model on a fixed batch has a constant Jacobian, so the own-step
  accumulation and the current reprojection coincide (no drift);
* closed forms of the cosine / relative-drift statistics and of the
  cancellation ratio (identical rows keep everything, opposite residuals
  cancel completely), and a brute-force loop for the ratio."""
import math

import numpy as np
import pytest

import oracle as O
from paper_2609_36738_gb300 import inputs as I
from tests import _indep as X

LINEAR_F32 = I.Workload("linear_probe_f32", 24, 16, (), 6, True, "f32", "uniform")
LAM, B1 = 0.5, 0.9


def _flat(ts):
    return np.concatenate([np.asarray(a).ravel() for a in ts])


def _own_step_trajectory(wl, steps, fixed_batch, lr=2e-2, seed=3):
    """Runs the own-step control (u = (1-lam) g + lam Mhat) for `steps` steps and
    records, per step, Mhat, h = Jbar^T qhat, qhat and s on that trajectory."""
    layers = X.oracle_layers(wl)
    params = X.params_f64(wl, I.init_params(wl, seed))
    M = [np.zeros_like(p) for p in params]
    v = [np.zeros_like(p) for p in params]
    q = np.zeros(wl.vocab)
    rec = []
    for t in range(1, steps + 1):
        xb, y = I.make_batch(wl, seed, 1 if fixed_batch else t)
        x = X.x_f64(wl, xb)
        out = O.bom_step(layers, wl.head_bias, params, x, y, q, t, lam=LAM, beta1=B1)
        q = out["q"]
        o, s, n_t = O.own_step_projection(layers, wl.head_bias, params, x, y)
        assert n_t == out["n_t"] and X.rel_l2(s, out["s"]) < 1e-15
        Mh = []
        for k in range(len(params)):
            M[k], mh = O.own_step_moment(M[k], o[k], t, B1)
            Mh.append(mh)
            params[k], v[k] = O.bom_update(params[k], O.mix_numerator(out["g"][k], mh, LAM), v[k], lr, 0.0, t)
        rec.append(dict(Mhat=Mh, h=out["h"], qhat=out["qhat"], s=s, o=o))
    return rec


def test_own_step_projection_equals_Jbar_s():
    """Jbar^T s_t with the per-example Jacobians by central differences."""
    wl = I.TINY_RAGGED_F32
    params = X.params_f64(wl, I.init_params(wl, 5))
    xb, y = I.make_batch(wl, 5, 1)
    x = X.x_f64(wl, xb)
    o, s, n_t = O.own_step_projection(X.oracle_layers(wl), wl.head_bias, params, x, y)
    J = X.fd_jacobians(wl, params, x)
    valid = y != I.IGNORE_INDEX
    Jbar = J[valid].sum(axis=0) / n_t        # batch mean over the supervised rows
    assert X.rel_l2(_flat(o), Jbar.T @ s) < 1e-7


def test_first_step_has_no_drift():
    """qhat_1 = s_1 and Mhat_1 = o_1, so Mhat_1 = h_1 on any model."""
    rec = _own_step_trajectory(I.TINY_RAGGED_F32, 1, fixed_batch=False)[0]
    assert X.rel_l2(_flat(rec["Mhat"]), _flat(rec["h"])) < 1e-13
    st = O.drift_statistics(rec["Mhat"], rec["h"])
    assert abs(st["cos"] - 1.0) < 1e-12 and st["rel"] < 1e-12


def test_classifier_bias_moment_equals_qhat():
    """Jbar_b = I on the head bias, so its Mhat_t is exactly qhat_t (and so is
    h_b) along a trajectory whose parameters and batches change."""
    rec = _own_step_trajectory(I.TINY_RAGGED_F32, 6, fixed_batch=False)
    for r in rec:
        assert X.rel_l2(r["Mhat"][-1], r["qhat"]) < 1e-13
        assert X.rel_l2(r["h"][-1], r["qhat"]) < 1e-13


def test_linear_model_on_a_fixed_batch_has_no_drift():
    """Constant Jacobian: own-step and current projections agree at every step."""
    rec = _own_step_trajectory(LINEAR_F32, 6, fixed_batch=True)
    for r in rec:
        st = O.drift_statistics(r["Mhat"], r["h"])
        assert st["rel"] < 1e-12 and abs(st["cos"] - 1.0) < 1e-12


def test_drift_appears_when_the_jacobian_moves():
    """Not vacuous: with a nonlinear backbone and changing batches the weight
    tensors drift, while the head bias still does not."""
    rec = _own_step_trajectory(I.TINY_RAGGED_F32, 6, fixed_batch=False)
    last = rec[-1]
    st = O.drift_statistics(last["Mhat"][:-1], last["h"][:-1])
    assert st["rel"] > 1e-3 and st["cos"] < 1.0 - 1e-6
    # sample replacement alone also drifts a linear model
    lin = _own_step_trajectory(LINEAR_F32, 6, fixed_batch=False)[-1]
    assert O.drift_statistics(lin["Mhat"][:1], lin["h"][:1])["rel"] > 1e-3


def test_drift_statistics_closed_forms():
    rng = np.random.default_rng(0)
    a = [rng.standard_normal((3, 4)), rng.standard_normal(5)]
    st = O.drift_statistics(a, a)
    assert abs(st["cos"] - 1) < 1e-15 and st["rel"] == 0.0
    st = O.drift_statistics(a, [-x for x in a])
    assert abs(st["cos"] + 1) < 1e-15 and abs(st["rel"] - 2) < 1e-15
    e1, e2 = [np.array([3.0, 0.0])], [np.array([0.0, 4.0])]
    st = O.drift_statistics(e1, e2)
    assert st["cos"] == 0.0 and abs(st["rel"] - 5.0 / 3.0) < 1e-15
    st2 = O.drift_statistics([7.0 * x for x in a], [0.5 * x for x in a])
    assert abs(st2["cos"] - 1) < 1e-15 and abs(st2["rel"] - (1 - 0.5 / 7.0)) < 1e-15


def _softmax_residuals(Z, y, valid):
    valid_idx = np.nonzero(valid)[0]
    R = np.zeros_like(Z)
    for i in valid_idx:
        R[i] = O.softmax_rows(Z[i:i + 1])[0]
        R[i, y[i]] -= 1.0
    return R


def test_cancellation_ratio_closed_forms():
    rng = np.random.default_rng(1)
    # identical rows: s = r_i, nothing cancels
    z = rng.standard_normal(9)
    Z = np.tile(z, (5, 1))
    y = np.full(5, 4)
    valid = np.ones(5, dtype=bool)
    ratio, _, _ = O.cancellation_ratio(_softmax_residuals(Z, y, valid), valid, 5)
    assert abs(ratio - 1.0) < 1e-14
    # two rows with equal logits and different labels: residuals cancel exactly
    Z2 = np.zeros((2, 2))
    y2 = np.array([0, 1])
    v2 = np.ones(2, dtype=bool)
    ratio, s_norm, mean_norm = O.cancellation_ratio(_softmax_residuals(Z2, y2, v2), v2, 2)
    assert ratio == 0.0 and abs(mean_norm - math.sqrt(0.5)) < 1e-15
    # duplicating the batch changes nothing; an ignored row is excluded
    Z3 = rng.standard_normal((7, 5))
    y3 = rng.integers(0, 5, 7)
    v3 = np.ones(7, dtype=bool)
    r_a = O.cancellation_ratio(_softmax_residuals(Z3, y3, v3), v3, 7)[0]
    Zd, yd, vd = np.vstack([Z3, Z3]), np.concatenate([y3, y3]), np.ones(14, dtype=bool)
    assert abs(O.cancellation_ratio(_softmax_residuals(Zd, yd, vd), vd, 14)[0] - r_a) < 1e-14
    Zi = np.vstack([Z3, rng.standard_normal((1, 5))])
    vi = np.concatenate([v3, [False]])
    yi = np.concatenate([y3, [0]])
    assert abs(O.cancellation_ratio(_softmax_residuals(Zi, yi, vi), vi, 7)[0] - r_a) < 1e-14
    assert 0.0 < r_a < 1.0


def test_cancellation_ratio_brute_force():
    rng = np.random.default_rng(2)
    n, c = 6, 4
    Z = rng.standard_normal((n, c))
    y = rng.integers(0, c, n)
    valid = np.ones(n, dtype=bool)
    R = O.residuals(Z, y, valid)
    # plain loops: softmax by hand, per-row Euclidean norms, the batch mean
    norms, mean = [], [0.0] * c
    for i in range(n):
        e = [math.exp(Z[i, j]) for j in range(c)]
        tot = sum(e)
        r = [e[j] / tot - (1.0 if j == y[i] else 0.0) for j in range(c)]
        norms.append(math.sqrt(sum(x * x for x in r)))
        for j in range(c):
            mean[j] += r[j] / n
    expect = math.sqrt(sum(x * x for x in mean)) / (sum(norms) / n)
    assert abs(O.cancellation_ratio(R, valid, n)[0] - expect) < 1e-14


def test_own_step_moment_closed_form():
    """M_t = (1-b1) sum_tau b1^(t-tau) o_tau; Mhat weights sum to one (Lemma 2)."""
    rng = np.random.default_rng(4)
    os_ = [rng.standard_normal(3) for _ in range(5)]
    M = np.zeros(3)
    for t, o in enumerate(os_, start=1):
        M, Mh = O.own_step_moment(M, o, t, B1)
        closed = sum((1 - B1) * B1 ** (t - k) * os_[k - 1] for k in range(1, t + 1))
        assert X.rel_l2(M, closed) < 1e-15
    same = [np.ones(3)] * 5
    M = np.zeros(3)
    for t, o in enumerate(same, start=1):
        M, Mh = O.own_step_moment(M, o, t, B1)
        assert np.allclose(Mh, 1.0, rtol=0, atol=1e-15)
    with pytest.raises(O.OracleError):
        O.own_step_moment(M, same[0], 0, B1)
