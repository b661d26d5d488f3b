"""Parity at the benchmark sizes, in the configuration bench.py times.

The fp64 oracle runs the full forward and the task-space pass (s_t, q_t,
qhat_t, CE, row log-sum-exp) on every row.  Where its full reverse pass would
take too long in fp64, it computes sampled rows of the head weight gradient
and of the head-input cotangent, and the tests check properties that hold at
any size: the vocabulary-column sums of u_W vanish (rows of R and qhat sum to
zero), and one backward of the mixed cotangent equals the mix of the two
separate passes, u = (1 - lambda) g + lambda h (Eq. mix-gradient)."""
import numpy as np
import pytest
import torch

import oracle as O
from paper_2609_36738_gb300 import bom as B
from paper_2609_36738_gb300 import inputs as I
from tests import _gpu as G
from tests import _indep as X

pytestmark = [pytest.mark.gpu, pytest.mark.slow]
TOL = G.TOL["bf16"]
LAM = 0.5


@pytest.fixture(scope="module", autouse=True)
def _built():
    G.ensure_built()


def _q0(V, seed=7):
    rng = np.random.default_rng(seed)
    q0 = (rng.standard_normal(V) * 0.01).astype(np.float32)
    return q0 - q0.mean(dtype=np.float64).astype(np.float32)


def _task_space(Z, y, q0, t):
    valid, n_t = O.supervised_set(y, Z.shape[1])
    R = O.residuals(Z, y, valid)
    s = O.batch_mean_residual(R, n_t)
    q, qhat = O.ema_update(q0.astype(np.float64), s, t, 0.9)
    ce, lse = O.cross_entropy(Z, y, valid, n_t)
    return dict(valid=valid, n_t=n_t, R=R, s=s, q=q, qhat=qhat, ce=ce, lse=lse)


def _check_task_space(gout, ref):
    st = gout["stats"]
    assert st["n_t"] == ref["n_t"]
    assert abs(st["loss"] - ref["ce"]) <= TOL * abs(ref["ce"])
    for k in ("s", "q", "qhat"):
        assert G.rel_l2(gout[k], ref[k]) < TOL, k
    v = ref["valid"]
    assert G.rel_l2(gout["lse"][v], ref["lse"][v]) < TOL
    assert abs(gout["s"].sum()) <= 1e-5 * np.abs(gout["s"]).sum() + 1e-7


def _sample(n, k, seed, extra=()):
    rng = np.random.default_rng(seed)
    return np.unique(np.concatenate([rng.integers(0, n, k), np.array(extra, dtype=np.int64)]))


def test_lm_output_block_full_size():
    """H 8192 x 768, head 50257 x 768, Zipf(1.1) labels: s_t, q_t, CE and lse on
    every row; u_W on 70 vocabulary rows; dH on 70 token rows."""
    wl = I.LM_HEAD_BF16
    params = I.init_params(wl, 0)
    x, y = I.make_batch(wl, 0, 1)
    t, q0 = 3, _q0(wl.vocab)
    gpu = G.GpuBom(wl, params)
    gpu.q.copy_(torch.from_numpy(q0))
    dx = torch.empty((wl.n_rows, wl.d_in), dtype=torch.bfloat16, device=G.DEV)
    B.bom_set_input_grad(gpu.model.h, dx)
    gout = gpu.step(x, y, t)
    u_w = G.np64(gout["grads"][0])

    H, W = I.bf16_to_f64(x), I.bf16_to_f64(params[0])
    Z = H @ W.T
    ref = _task_space(Z, y, q0, t)
    del Z
    _check_task_space(gout, ref)
    rv = _sample(wl.vocab, 64, 1, extra=(0, 1, 2, wl.vocab - 1))
    gw = O.head_weight_grad_rows(ref["R"], H, ref["valid"], ref["qhat"], ref["n_t"], LAM, rv)
    assert G.rel_l2(u_w[rv], gw) < TOL
    ri = _sample(wl.n_rows, 64, 2, extra=(0, wl.n_rows - 1))
    gi = O.head_input_grad_rows(ref["R"], W, ref["valid"], ref["qhat"], ref["n_t"], LAM, ri)
    assert G.rel_l2(G.np64(dx)[ri], gi) < TOL
    # rows of R and qhat sum to zero, so the vocabulary-column sums of u_W vanish
    assert np.abs(u_w.sum(axis=0)).max() <= 2e-2 * np.abs(u_w).sum(axis=0).max()


def test_lm_block_with_swiglu_mlps_full_size():
    """16384 tokens, two SwiGLU MLPs (d 2048, ffn 8192), head 32000 x 2048:
    s_t, q_t, CE, lse on every row (fp64 forward), u_W of the head on sampled
    rows, and u = (1-lambda) g + lambda h for every tensor."""
    wl = I.LM_MLP_BF16
    params = I.init_params(wl, 0)
    x, y = I.make_batch(wl, 0, 1)
    t, q0 = 2, _q0(wl.vocab)
    gpu = G.GpuBom(wl, params)
    gpu.q.copy_(torch.from_numpy(q0))
    gout = gpu.step(x, y, t)
    grads_u = [G.np64(g) for g in gout["grads"]]
    del gout["grads"]

    gh = G.GpuBom(wl, params, out_mode=B.BOM_OUT_G_AND_H)
    gh.q.copy_(torch.from_numpy(q0))
    o2 = gh.step(x, y, t)
    for k, u in enumerate(grads_u):
        mix = (1 - LAM) * G.np64(o2["grads"][k]) + LAM * G.np64(o2["h"][k])
        assert G.rel_l2(u, mix) < TOL, k
    del o2, gh

    p64 = X.params_f64(wl, params)
    Z, saved = O.forward(X.oracle_layers(wl), False, p64, I.bf16_to_f64(x))
    ref = _task_space(Z, y, q0, t)
    del Z
    _check_task_space(gout, ref)
    h_last = saved[1]
    rv = _sample(wl.vocab, 64, 3, extra=(0, 1, 2, wl.vocab - 1))
    gw = O.head_weight_grad_rows(ref["R"], h_last, ref["valid"], ref["qhat"], ref["n_t"], LAM, rv)
    u_head = grads_u[-1]
    assert G.rel_l2(u_head[rv], gw) < TOL
    assert np.abs(u_head.sum(axis=0)).max() <= 2e-2 * np.abs(u_head).sum(axis=0).max()


def test_vision_head_twenty_steps_full_size():
    """768 -> 3072 -> 768 -> 1000 classes, batch 256, bf16: 20 BOM steps, each
    followed by the update of every tensor.  Every step is checked on the same
    inputs the GPU step read (its bf16 parameters and q_{t-1}); the oracle also
    runs its own fp64 trajectory, and the final master weights of the two
    trajectories must agree."""
    wl = I.VISION_HEAD_BF16
    lr, b2, eps = 1e-3, 0.999, 1e-8
    F = lambda v: float(np.float32(v))
    wds = I.weight_decay_mask(wl, 0.01)
    params = I.init_params(wl, seed=11)
    p64 = X.params_f64(wl, params)
    gpu = G.GpuBom(wl, params)
    master = [torch.from_numpy(I.bf16_to_f32(p)).to(G.DEV) for p in params]
    vs = [torch.zeros(p.shape, dtype=torch.float32, device=G.DEV) for p in params]
    vo = [np.zeros(p.shape) for p in p64]
    q = np.zeros(wl.vocab)
    worst = 0.0
    for t in range(1, wl.steps + 1):
        xb, y = I.make_batch(wl, seed=11, step=t)
        p_in = [G.np64(p) for p in gpu.params]
        q_in = G.np64(gpu.q)
        gout = gpu.step(xb, y, t)
        same = G.oracle_step(wl, p_in, xb, y, q_in, t)
        assert gout["stats"]["n_t"] == same["n_t"]
        assert G.rel_l2(gout["q"], same["q"]) < TOL
        for k in range(len(params)):
            err = G.rel_l2(G.np64(gout["grads"][k]), same["u"][k])
            worst = max(worst, err)
            assert err < TOL, (t, k, err)
            B.bom_update(master[k], gout["grads"][k], B.BOM_BF16, None, vs[k], gpu.params[k], master[k].numel(),
                         lr, wds[k], 0.5, b2, eps, t)
        # the oracle's own trajectory computes with bf16 copies of its fp64
        # master weights, as the GPU does with its fp32 ones (bf16 autocast)
        oref = G.oracle_step(wl, [G.bf16_round(p) for p in p64], xb, y, q, t)
        q = oref["q"]
        for k in range(len(params)):
            p64[k], vo[k] = O.bom_update(p64[k], oref["u"][k], vo[k], F(lr), F(wds[k]), t, F(b2), F(eps))
        torch.cuda.synchronize()
    print(f"vision head, 20 steps: worst per-step relative L2 of u {worst:.3e}")
    for k in range(len(params)):
        assert G.rel_l2(G.np64(master[k]), p64[k]) < TOL
