"""Pins of the fp64 oracle against facts the paper and mathematics fix.

None of these compare the oracle with itself: the references are central
finite-difference Jacobians of an independent torch forward, torch autograd,
torch.optim.AdamW, closed forms, and numbers printed in the paper
(tests/golden/paper_coefficients.json, each with its citation).
"""
import json
import math
import os

import numpy as np
import pytest
import torch

import oracle as O
from paper_2609_36738_gb300 import inputs as I
from tests import _indep as X

GOLDEN = json.load(open(os.path.join(os.path.dirname(__file__), "golden", "paper_coefficients.json")))
FIXED = GOLDEN["fixed_coefficients"]


def _setup(wl, seed=0, t=3, bias_scale=0.1, zero_sum_q=True):
    params = X.params_f64(wl, I.init_params(wl, seed))
    g = np.random.default_rng(seed + 77)
    # non-zero biases so that every parameter path carries signal
    for k, (name, shape, is_mat) in enumerate(wl.param_shapes()):
        if not is_mat:
            params[k] = params[k] + bias_scale * g.standard_normal(shape)
    xb, y = I.make_batch(wl, seed, 1)
    x = X.x_f64(wl, xb)
    q_prev = 0.05 * g.standard_normal(wl.vocab)
    if zero_sum_q:
        q_prev -= q_prev.mean()
    return params, x, y, q_prev, t


@pytest.fixture(scope="module")
def tiny_jac():
    """Step at t = 3 on the 64-128-10 GELU MLP (P = 9,610, N = 32) with the
    per-example Jacobians of every logit by central differences."""
    wl = I.TINY_MLP_F32
    params, x, y, q_prev, t = _setup(wl)
    out = O.bom_step(X.oracle_layers(wl), wl.head_bias, params, x, y, q_prev, t,
                     lam=0.5, beta1=0.9)
    J = X.fd_jacobians(wl, params, x)
    return wl, params, x, y, q_prev, t, out, J


def _flat(ts):
    return np.concatenate([np.asarray(a).ravel() for a in ts])


def test_param_count_matches_tiny_config():
    assert I.TINY_MLP_F32.n_params() == 9610
    assert I.VISION_HEAD_BF16.n_params() == 5_491_432
    assert I.LM_MLP_BF16.n_params() == 166_199_296


def test_forward_matches_independent_torch():
    for wl in (I.TINY_MLP_F32, I.TINY_RAGGED_F32, I.VISION_SMALL, I.LM_MLP_SMALL, I.TINY_NORM_F32, I.LM_NORM_SMALL):
        params, x, y, _, _ = _setup(wl)
        Z, _ = O.forward(X.oracle_layers(wl), wl.head_bias, params, x)
        Zt = X.torch_forward(wl, [torch.tensor(p) for p in params], torch.tensor(x)).numpy()
        assert X.rel_l2(Z, Zt) < 1e-13


def test_batch_decomposition_g_equals_Jbar_s_plus_c(tiny_jac):
    """Eq. batch-decomposition: g = Jbar^T s + c, with J_i by finite differences."""
    wl, params, x, y, q_prev, t, out, J = tiny_jac
    R, s, n = out["R"], out["s"], out["n_t"]
    Jbar = J.mean(axis=0)
    c = np.einsum("ncp,nc->p", J - Jbar, R - s) / n
    direct = np.einsum("ncp,nc->p", J, R) / n
    g = _flat(out["g"])
    assert X.rel_l2(Jbar.T @ s + c, direct) < 1e-12     # the identity itself
    assert X.rel_l2(g, direct) < 1e-7                   # oracle's reverse pass


def test_reprojection_h_equals_Jbar_qhat(tiny_jac):
    """h_t = Jbar_t^T qhat_t (Eq. drift-telemetry), Jbar by finite differences."""
    wl, params, x, y, q_prev, t, out, J = tiny_jac
    Jbar = J.mean(axis=0)
    assert X.rel_l2(_flat(out["h"]), Jbar.T @ out["qhat"]) < 1e-7


def test_u_is_mix_of_g_and_h_and_matches_decomposition(tiny_jac):
    """Eq. mix-gradient, and u = (1-lam)(Jbar^T s + c) + lam Jbar^T qhat."""
    wl, params, x, y, q_prev, t, out, J = tiny_jac
    lam = 0.5
    Jbar = J.mean(axis=0)
    R, s, n = out["R"], out["s"], out["n_t"]
    c = np.einsum("ncp,nc->p", J - Jbar, R - s) / n
    u = _flat(out["u"])
    assert X.rel_l2(u, (1 - lam) * _flat(out["g"]) + lam * _flat(out["h"])) < 1e-14
    assert X.rel_l2(u, (1 - lam) * (Jbar.T @ s + c) + lam * Jbar.T @ out["qhat"]) < 1e-7


def test_u_decomposition_weights_printed_in_paper(tiny_jac):
    """Eq. u-decomposition at lambda = 0.5, beta1 = 0.9 once bias correction is
    negligible: u = 0.55 Jbar^T s + 0.5 c + 0.45 Jbar^T q_{t-1}."""
    wl, params, x, y, q_prev, _, _, J = tiny_jac
    gw = GOLDEN["u_decomposition_weights"]
    lam, b1 = gw["lambda"], gw["beta1"]
    t = 400                                              # beta1^t ~ 5e-19
    out = O.bom_step(X.oracle_layers(wl), wl.head_bias, params, x, y, q_prev, t, lam=lam, beta1=b1)
    Jbar = J.mean(axis=0)
    R, s, n = out["R"], out["s"], out["n_t"]
    c = np.einsum("ncp,nc->p", J - Jbar, R - s) / n
    pred = (gw["current_batch_mean_weight"] * Jbar.T @ s + gw["covariance_weight"] * c
            + gw["history_weight"] * Jbar.T @ q_prev)
    assert X.rel_l2(_flat(out["u"]), pred) < 1e-7
    # the printed weights are the closed-form coefficients of that equation
    assert math.isclose((1 - lam) + lam * (1 - b1), gw["current_batch_mean_weight"], abs_tol=1e-15)
    assert math.isclose(lam * b1, gw["history_weight"], abs_tol=1e-15)
    aw = GOLDEN["adamw_first_moment_weights"]
    assert math.isclose(1 - aw["beta1"], aw["current_weight"], abs_tol=1e-15)


@pytest.mark.parametrize("name", ["tiny_mlp_f32", "tiny_ragged_f32", "vision_small", "lm_mlp_small",
                                  "lm_head_small", "tiny_norm_f32", "lm_norm_small"])
def test_u_matches_autograd_of_mix_objective(name):
    """One backward of L_mix (Eq. mix-objective) through torch autograd (the
    RMSNorm workloads go through torch.nn.functional.rms_norm)."""
    wl = I.WORKLOADS[name]
    params, x, y, q_prev, t = _setup(wl, seed=1)
    out = O.bom_step(X.oracle_layers(wl), wl.head_bias, params, x, y, q_prev, t, lam=0.5, beta1=0.9)
    grads, ce = X.autograd_mix(wl, params, x, y, out["qhat"], 0.5)
    for a, b in zip(out["u"], grads):
        assert a.shape == b.shape
        assert X.rel_l2(a, b) < 1e-12
    assert math.isclose(out["ce"], ce, rel_tol=1e-13)
    assert X.rel_l2(out["dX_u"], X.autograd_mix.last_dX) < 1e-12      # input cotangent
    g_grads, _ = X.autograd_mix(wl, params, x, y, out["qhat"], 0.0)
    for a, b in zip(out["g"], g_grads):
        assert X.rel_l2(a, b) < 1e-12


def test_output_bias_closed_form(tiny_jac):
    """Jbar_b = I for the classifier bias: g_b = s, h_b = qhat (historical-projection
    control appendix), so u_b = (1-lam) s + lam qhat."""
    wl, params, x, y, q_prev, t, out, J = tiny_jac
    assert np.allclose(out["g"][-1], out["s"], rtol=0, atol=1e-15)
    assert np.allclose(out["h"][-1], out["qhat"], rtol=0, atol=1e-15)
    assert np.allclose(out["u"][-1], 0.5 * out["s"] + 0.5 * out["qhat"], rtol=0, atol=1e-15)


def test_zero_sum_invariant():
    """Residual coordinates sum to zero, hence so do s_t and q_t (Section 3.1)."""
    for wl in (I.TINY_MLP_F32, I.LM_HEAD_SMALL, I.VISION_SMALL):
        params, x, y, q_prev, t = _setup(wl, seed=2)
        out = O.bom_step(X.oracle_layers(wl), wl.head_bias, params, x, y, q_prev, t)
        assert abs(out["s"].sum()) <= 1e-14 * (1 + np.abs(out["s"]).sum())
        assert abs(out["q"].sum()) <= 1e-14 * (1 + np.abs(out["q"]).sum())
        assert np.abs(out["R"].sum(axis=1)).max() < 1e-14


def test_binary_softmax_history_is_one_scalar():
    """C = 2: q_t = (a_t, -a_t) and Jbar^T qhat = ahat grad_theta mean(z_1 - z_2)
    (Section 3.1, 'How small the stored history is')."""
    wl = I.Workload("binary", 16, 5, (I.Layer(I.LINEAR_GELU, 5, 6, True),), 2, True, "f32", "uniform")
    params, x, y, _, _ = _setup(wl, seed=3)
    layers = X.oracle_layers(wl)
    q = np.zeros(2)
    for t in range(1, 5):
        xb, y = I.make_batch(wl, 3, t)
        out = O.bom_step(layers, True, params, X.x_f64(wl, xb), y, q, t)
        q = out["q"]
        assert abs(q[0] + q[1]) < 1e-16
    J = X.fd_jacobians(wl, params, X.x_f64(wl, xb))
    margin_grad = (J[:, 0, :] - J[:, 1, :]).mean(axis=0)
    assert X.rel_l2(_flat(out["h"]), out["qhat"][0] * margin_grad) < 1e-7


def test_ema_closed_form_and_lemma2_weights():
    """q_t = sum_tau (1-b1) b1^(t-tau) s_tau; the bias-corrected weights
    alpha_{t,tau} = (1-b1) b1^(t-tau) / (1-b1^t) sum to one (Lemma 2)."""
    g = np.random.default_rng(5)
    for b1 in (0.9, 0.5, 0.99):
        T = 7
        S = g.standard_normal((T, 11))
        q = np.zeros(11)
        for t in range(1, T + 1):
            q, qhat = O.ema_update(q, S[t - 1], t, b1)
            w = np.array([(1 - b1) * b1 ** (t - tau) for tau in range(1, t + 1)])
            assert np.allclose(q, w @ S[:t], rtol=0, atol=1e-15)
            alpha = w / (1 - b1 ** t)
            assert abs(alpha.sum() - 1.0) < 1e-14
            assert np.allclose(qhat, alpha @ S[:t], rtol=0, atol=1e-14)
        # constant signal: the bias-corrected EMA is that signal
        q = np.zeros(11)
        for t in range(1, T + 1):
            q, qhat = O.ema_update(q, S[0], t, b1)
        assert np.allclose(qhat, S[0], rtol=0, atol=1e-14)


def test_beta1_zero_gives_qhat_equal_s():
    """beta1 = 0: the task-space history is the current s_t (beta1 sweep, qhat = s)."""
    wl = I.LM_HEAD_SMALL
    params, x, y, q_prev, t = _setup(wl, seed=4)
    out = O.bom_step(X.oracle_layers(wl), wl.head_bias, params, x, y, q_prev, t, beta1=0.0)
    assert np.array_equal(out["qhat"], out["s"])


def test_lambda_zero_is_adamw_with_beta1_zero():
    """lambda = 0 reduces u to the CE gradient, and the update to AdamW with
    beta1 = 0 (torch.optim.AdamW, fp64)."""
    wl = I.TINY_RAGGED_F32
    layers = X.oracle_layers(wl)
    params, _, _, _, _ = _setup(wl, seed=6)
    lr, wd = 1e-2, FIXED["omega"]
    wds = I.weight_decay_mask(wl, wd)
    tp = [torch.tensor(p.copy(), requires_grad=True) for p in params]
    groups = [{"params": [p], "weight_decay": w} for p, w in zip(tp, wds)]
    opt = torch.optim.AdamW(groups, lr=lr, betas=(0.0, FIXED["beta2"]), eps=FIXED["eps"],
                            foreach=False, fused=False)
    v = [np.zeros_like(p) for p in params]
    q = np.zeros(wl.vocab)
    for t in range(1, 4):
        xb, y = I.make_batch(wl, 6, t)
        xx = X.x_f64(wl, xb)
        out = O.bom_step(layers, wl.head_bias, params, xx, y, q, t, lam=0.0)
        q = out["q"]
        ag, _ = X.autograd_mix(wl, params, xx, y, out["qhat"], 0.0)
        for a, b in zip(out["u"], ag):
            assert X.rel_l2(a, b) < 1e-12
        new = []
        for k, p in enumerate(params):
            th, v[k] = O.bom_update(p, out["u"][k], v[k], lr, wds[k], t, FIXED["beta2"], FIXED["eps"])
            new.append(th)
        params = new
        for p, gr in zip(tp, ag):
            p.grad = torch.tensor(gr)
        opt.step()
        for a, p in zip(params, tp):
            assert X.rel_l2(a, p.detach().numpy()) < 1e-14


def test_update_first_step_closed_form():
    """t = 1, omega = 0: v = (1-b2) u^2, vhat = u^2, so delta = -eta u / (|u| + eps)."""
    g = np.random.default_rng(8)
    th = g.standard_normal(1000)
    u = g.standard_normal(1000) * 1e-3
    new, v = O.bom_update(th, u, np.zeros(1000), 1e-3, 0.0, 1)
    assert np.allclose(new - th, -1e-3 * u / (np.abs(u) + 1e-8), rtol=1e-12, atol=0)
    assert np.allclose(v, (1 - 0.999) * u * u, rtol=1e-15, atol=0)


def test_update_decoupled_decay_acts_on_old_theta():
    """u = 0: theta <- (1 - eta omega) theta exactly."""
    th = np.linspace(-2, 2, 9)
    new, _ = O.bom_update(th, np.zeros(9), np.zeros(9), 0.1, 0.01, 5)
    assert np.array_equal(new, (1 - 0.1 * 0.01) * th)


def test_ignored_rows_are_excluded_from_every_mean():
    """I_t excludes ignored targets from both averages (LM construction appendix):
    a batch with ignored rows equals the batch restricted to its valid rows."""
    wl = I.LM_MLP_SMALL
    params, x, y, q_prev, t = _setup(wl, seed=9)
    assert (y == I.IGNORE_INDEX).sum() > 0
    layers = X.oracle_layers(wl)
    a = O.bom_step(layers, wl.head_bias, params, x, y, q_prev, t)
    keep = y != I.IGNORE_INDEX
    b = O.bom_step(layers, wl.head_bias, params, x[keep], y[keep], q_prev, t)
    assert a["n_t"] == int(keep.sum()) == b["n_t"]
    for key in ("s", "q", "qhat"):
        assert X.rel_l2(a[key], b[key]) < 1e-14
    for ga, gb in zip(a["u"], b["u"]):
        assert X.rel_l2(ga, gb) < 1e-12
    assert math.isclose(a["ce"], b["ce"], rel_tol=1e-13)
    # the label histogram inside s is exact: s + counts / N_t = mean softmax
    counts = np.bincount(y[keep], minlength=wl.vocab)
    P = O.softmax_rows(a["Z"])[keep]
    assert np.allclose(a["s"] + counts / a["n_t"], P.sum(0) / a["n_t"], rtol=0, atol=1e-15)


def test_error_cases():
    wl = I.LM_HEAD_SMALL
    params, x, y, q_prev, t = _setup(wl, seed=10)
    layers = X.oracle_layers(wl)
    bad = y.copy()
    bad[3] = wl.vocab
    with pytest.raises(O.LabelError):
        O.bom_step(layers, False, params, x, bad, q_prev, t)
    bad[3] = -1
    with pytest.raises(O.LabelError):
        O.bom_step(layers, False, params, x, bad, q_prev, t)
    with pytest.raises(O.EmptyError):
        O.bom_step(layers, False, params, x, np.full_like(y, I.IGNORE_INDEX), q_prev, t)
    with pytest.raises(O.OracleError):
        O.bom_step(layers, False, params, x, y, q_prev, 0)


def test_softmax_and_ce_brute_force():
    """Softmax, log-sum-exp and CE against plain Python loops."""
    g = np.random.default_rng(11)
    Z = g.standard_normal((5, 7)) * 3
    y = np.array([0, 6, 3, 3, 1], dtype=np.int32)
    P = O.softmax_rows(Z)
    lse = O.log_sum_exp_rows(Z)
    valid, n = O.supervised_set(y, 7)
    ce, _ = O.cross_entropy(Z, y, valid, n)
    tot = 0.0
    for i in range(5):
        den = sum(math.exp(Z[i, k]) for k in range(7))
        assert math.isclose(lse[i], math.log(den), rel_tol=1e-14)
        for k in range(7):
            assert math.isclose(P[i, k], math.exp(Z[i, k]) / den, rel_tol=1e-13)
        tot += math.log(den) - Z[i, y[i]]
    assert math.isclose(ce, tot / 5, rel_tol=1e-14)
    # shift invariance keeps large logits finite
    assert np.allclose(O.softmax_rows(Z + 1000.0), P, rtol=1e-12, atol=0)
    R = O.residuals(Z, y, valid)
    for i in range(5):
        for k in range(7):
            assert math.isclose(R[i, k], P[i, k] - (1.0 if k == y[i] else 0.0), abs_tol=1e-15)


def test_checkpoint_accounting_matches_state_layout():
    """fp32 theta + v is 8 bytes per parameter versus AdamW's 12 (theta, m, v)."""
    ck = GOLDEN["checkpoint_bytes_per_parameter"]
    bom_state = ["theta", "v"]        # q is d_out-sized, not parameter-shaped
    assert 4 * len(bom_state) == ck["bom"]
    assert 4 * (len(bom_state) + 1) == ck["adamw"]
