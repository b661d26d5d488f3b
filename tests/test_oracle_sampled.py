"""The oracle's sampled head-gradient helpers equal the rows of its full
reverse pass (they restate the same formulas on a subset of rows)."""
import numpy as np
import pytest

import oracle as O
import oracle.bom_oracle as OM
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


def _all_rows_case(name, seed):
    wl = I.WORKLOADS[name]
    params = X.params_f64(wl, I.init_params(wl, seed))
    xb, y = I.make_batch(wl, seed, 1)
    x = X.x_f64(wl, xb)
    q0 = np.random.default_rng(seed + 1).standard_normal(wl.vocab) * 0.01
    layers = X.oracle_layers(wl)
    out = O.bom_step(layers, wl.head_bias, params, x, y, q0, 3)
    _, saved = O.forward(layers, wl.head_bias, params, x)
    return wl, params, x, y, layers, out, saved


@pytest.mark.parametrize("name", ["lm_mlp_small", "lm_mlp_mid", "lm_norm_small", "vision_small",
                                  "tiny_ragged_f32", "tiny_norm_f32", "lm_head_small"])
def test_sampled_rows_of_every_tensor_match_full_backward(name):
    """mix_grad_rows on sampled rows (first, last and interior rows of every
    tensor) equals the same rows of the oracle's full reverse pass of L_mix."""
    wl, params, x, y, layers, out, saved = _all_rows_case(name, 5)
    rng = np.random.default_rng(9)
    rows = []
    for p in params:
        n = p.shape[0]
        rows.append(np.unique(np.concatenate([[0, n - 1], rng.integers(0, n, 6)])))
    got = O.mix_grad_rows(layers, wl.head_bias, params, saved, out["R"], out["valid"], out["qhat"], out["n_t"],
                          0.5, rows)
    for k, p in enumerate(params):
        assert got[k].shape == ((len(rows[k]),) + p.shape[1:]), k
        assert X.rel_l2(got[k], out["u"][k][rows[k]]) < 1e-12, (name, k)


@pytest.mark.parametrize("name", ["lm_mlp_small", "vision_small", "lm_norm_small"])
def test_sampled_rows_match_torch_autograd(name):
    """The same rows against torch autograd of L_mix (an implementation that
    shares nothing with the oracle): every row of every tensor."""
    wl, params, x, y, layers, out, saved = _all_rows_case(name, 6)
    rows = [np.arange(p.shape[0]) for p in params]
    got = O.mix_grad_rows(layers, wl.head_bias, params, saved, out["R"], out["valid"], out["qhat"], out["n_t"],
                          0.5, rows)
    ref, _ = X.autograd_mix(wl, params, x, y, out["qhat"], 0.5)
    for k in range(len(params)):
        assert X.rel_l2(got[k], ref[k]) < 1e-11, (name, k)


def test_sampled_rows_reject_plausible_mistakes():
    """A restatement that drops the residual path of a SwiGLU sublayer, or
    uses SiLU in place of SiLU', no longer matches the full reverse pass."""
    wl, params, x, y, layers, out, saved = _all_rows_case("lm_mlp_small", 7)
    rows = [np.arange(min(p.shape[0], 16)) for p in params]
    good = O.mix_grad_rows(layers, wl.head_bias, params, saved, out["R"], out["valid"], out["qhat"], out["n_t"],
                           0.5, rows)
    for mutate in ("no_residual", "silu_for_silu_prime"):
        orig = (OM.silu_prime, OM.silu)
        tape, h_last = saved
        if mutate == "silu_for_silu_prime":
            OM.silu_prime = OM.silu
            bad_saved = saved
        else:
            # x + A W_d^T without the skip path: the lower layer sees dy only through W_d
            bad_tape = [(k, np.zeros_like(xx), G, U, A) if k == "swiglu" and li == 0 else (k, xx, G, U, A)
                        for li, (k, xx, G, U, A) in enumerate(tape)]
            bad_saved = (bad_tape, h_last)
        try:
            bad = O.mix_grad_rows(layers, wl.head_bias, params, bad_saved, out["R"], out["valid"], out["qhat"],
                                  out["n_t"], 0.5, rows)
        finally:
            OM.silu_prime, OM.silu = orig
        worst = max(X.rel_l2(b, out["u"][k][rows[k]]) for k, b in enumerate(bad))
        assert worst > 1e-3, mutate
    assert max(X.rel_l2(g, out["u"][k][rows[k]]) for k, g in enumerate(good)) < 1e-12
