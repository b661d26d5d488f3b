"""The seeded input generator follows the recipe the design states: the
stand-ins for the paper's workloads (no dataset is available) are
- X ~ N(0, 1);
- weight matrices Kaiming-uniform U(-sqrt(6/fan_in), +sqrt(6/fan_in)), the LM
  head N(0, 0.02), biases 0, RMSNorm weights 1 + N(0, 0.1^2);
- labels uniform over the classes, or Zipf(1.1) over the vocabulary (rank k ->
  token k - 1, truncated at V) for the LM settings;
- a stated fraction of rows carrying the ignore index;
- the same seed giving the same bytes, each step its own batch.
Statistical checks use tolerances of several standard errors."""
import numpy as np
import pytest

from paper_2609_36738_gb300 import inputs as I


def _f64(a, wl):
    return I.bf16_to_f64(a) if wl.dtype == "bf16" else a.astype(np.float64)


@pytest.mark.parametrize("name", ["vision_head_bf16", "lm_mlp_small", "tiny_mlp_f32", "lm_norm_small"])
def test_parameter_initialisation(name):
    wl = I.WORKLOADS[name]
    params = I.init_params(wl, seed=3)
    for (pname, shape, is_mat), p in zip(wl.param_shapes(), params):
        v = _f64(p, wl)
        assert v.shape == tuple(shape)
        if pname.endswith("norm_weight"):
            assert abs(v.mean() - 1.0) < 5 * 0.1 / np.sqrt(v.size) + 0.01
            assert abs(v.std() - 0.1) < 0.02
        elif not is_mat:
            assert not v.any(), pname        # biases start at zero
        elif pname.startswith("head") and wl.head_init == "normal002":
            assert abs(v.std() - 0.02) < 0.02 * 0.05, pname
            assert abs(v.mean()) < 5 * 0.02 / np.sqrt(v.size)
        else:
            bound = np.sqrt(6.0 / shape[1])
            # bf16 rounding may lift a value by at most half a unit in the last place
            assert np.abs(v).max() <= bound * (1 + 2.0 ** -8), pname
            assert abs(v.std() - bound / np.sqrt(3.0)) < 0.05 * bound / np.sqrt(3.0), pname


def test_inputs_are_standard_normal():
    wl = I.LM_MLP_SMALL
    x, _ = I.make_batch(wl, seed=4, step=1)
    v = _f64(x, wl)
    assert abs(v.mean()) < 5 / np.sqrt(v.size) + 0.01
    assert abs(v.std() - 1.0) < 0.02


def test_zipf_labels_follow_the_truncated_law():
    vocab, n, a = 1000, 200_000, 1.1
    y = I.zipf_labels(np.random.default_rng(5), n, vocab, a)
    assert y.min() >= 0 and y.max() < vocab
    ranks = np.arange(1, vocab + 1, dtype=np.float64)
    pmf = ranks ** -a / np.sum(ranks ** -a)
    freq = np.bincount(y, minlength=vocab) / n
    for k in range(10):                      # the head of the law, where the mass is
        se = np.sqrt(pmf[k] * (1 - pmf[k]) / n)
        assert abs(freq[k] - pmf[k]) < 5 * se, k
    assert abs(freq[100:].sum() - pmf[100:].sum()) < 5 * np.sqrt(pmf[100:].sum() / n)


def test_uniform_labels_and_the_ignore_fraction():
    wl = I.WORKLOADS["lm_head_small"]            # Zipf labels, 10% ignored
    ys = np.concatenate([I.make_batch(wl, seed=6, step=t)[1] for t in range(1, 41)])
    frac = np.mean(ys == I.IGNORE_INDEX)
    assert abs(frac - wl.ignore_frac) < 5 * np.sqrt(wl.ignore_frac * (1 - wl.ignore_frac) / ys.size)
    kept = ys[ys != I.IGNORE_INDEX]
    assert kept.min() >= 0 and kept.max() < wl.vocab
    wl = I.VISION_HEAD_BF16                       # uniform over 1000 classes, none ignored
    ys = np.concatenate([I.make_batch(wl, seed=7, step=t)[1] for t in range(1, 21)])
    assert (ys >= 0).all() and (ys < wl.vocab).all()
    counts = np.bincount(ys, minlength=wl.vocab)
    exp = ys.size / wl.vocab
    chi2 = ((counts - exp) ** 2 / exp).sum()
    assert chi2 < wl.vocab + 5 * np.sqrt(2 * wl.vocab)


def test_seeds_and_steps():
    wl = I.VISION_SMALL
    a = I.make_batch(wl, seed=8, step=2)
    b = I.make_batch(wl, seed=8, step=2)
    c = I.make_batch(wl, seed=8, step=3)
    assert np.array_equal(a[0], b[0]) and np.array_equal(a[1], b[1])
    assert not np.array_equal(a[0], c[0])
    p = I.init_params(wl, seed=8)
    q = I.init_params(wl, seed=8)
    assert all(np.array_equal(u, v) for u, v in zip(p, q))


def test_weight_decay_applies_to_matrices_only():
    wl = I.LM_NORM_SMALL
    wd = I.weight_decay_mask(wl, 0.1)
    for (_, _, is_mat), w in zip(wl.param_shapes(), wd):
        assert w == (0.1 if is_mat else 0.0)
