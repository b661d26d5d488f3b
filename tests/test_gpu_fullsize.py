"""Parity at the benchmark sizes, in the configuration bench.py times.

The fp64 oracle runs the full forward and the task-space pass (s_t, q_t,
qhat_t, CE, row log-sum-exp) on every row.  Where its full reverse pass would
take too long in fp64, it restates that pass for sampled output rows of every
weight gradient (every cotangent is still formed over all rows), and the
tests also check properties that hold at any size: the vocabulary-column sums
of u_W vanish (rows of R and qhat sum to zero), and one backward of the mixed
cotangent equals the mix of the two separate passes, u = (1 - lambda) g +
lambda h (Eq. mix-gradient)."""
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


def _outputs(model, wl):
    qp, sp, lp = model.outputs()
    return {"qhat": G.host_f32(qp, wl.vocab), "s": G.host_f32(sp, wl.vocab), "lse": G.host_f32(lp, wl.n_rows)}


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


def _dev_rows(t, rows):
    """float64 host copy of rows `rows` (first index) of a device tensor."""
    return G.np64(t.index_select(0, torch.from_numpy(np.asarray(rows, dtype=np.int64)).to(t.device)))


def test_lm_block_with_swiglu_mlps_full_size():
    """16384 tokens, two SwiGLU MLPs (d 2048, ffn 8192), head 32000 x 2048, in
    the launch configuration bench.py times: the BOM-AdamW update fused into
    the step (lr 1e-4, weight decay 0.1 on the matrices), one batch repeated.
    Two fused steps move the state; at t = 3 the fp64 oracle runs on the inputs
    that step reads (bf16 parameters, q_2, theta and v) and checks
      - s_t, q_t, qhat_t, CE and lse on every row, N_t exactly;
      - u of all seven tensors on sampled rows (a second handle writes u from
        the same inputs; Eq. mix-gradient through the head and both
        sublayers);
      - theta and v of the fused step on the same rows (Section 3.4);
      - u = (1 - lambda) g + lambda h for every tensor (a G_AND_H handle)."""
    wl = I.LM_MLP_BF16
    lr, wd_mat, b2, eps, t_chk = 1e-4, 0.1, 0.999, 1e-8, 3
    F = lambda v: float(np.float32(v))
    wds = I.weight_decay_mask(wl, wd_mat)
    params = I.init_params(wl, 0)
    x, y = I.make_batch(wl, 0, 1)
    fz = G.GpuBom(wl, params)
    theta = [torch.from_numpy(I.bf16_to_f32(p)).to(G.DEV) for p in params]
    v = [torch.zeros(p.shape, dtype=torch.float32, device=G.DEV) for p in params]
    B.bom_set_fused_update(fz.model.h, theta, v, wds, lr, b2, eps)
    xd = G.to_dev(x)
    yd = torch.from_numpy(np.ascontiguousarray(y, dtype=np.int32)).to(G.DEV)
    for t in range(1, t_chk):
        fz.model.step(xd, yd, wl.n_rows, fz.params, fz.q, t, None, None)
        assert fz.model.stats()["code"] == B.BOM_OK

    # the inputs of step t_chk, as the fused step will read them
    p_in = [p.clone() for p in fz.params]
    q_in = G.np64(fz.q)
    rng = np.random.default_rng(3)
    rows = [np.unique(np.concatenate([rng.integers(0, p.shape[0], 64), [0, p.shape[0] - 1]])) for p in params]
    th_in = [_dev_rows(a, r) for a, r in zip(theta, rows)]
    v_in = [_dev_rows(a, r) for a, r in zip(v, rows)]

    # u from the same inputs on a handle that writes it
    us = G.GpuBom(wl, p_in)
    us.q.copy_(fz.q)
    gout = us.step(x, y, t_chk)
    u_rows = [_dev_rows(g, r) for g, r in zip(gout["grads"], rows)]
    # g and h on a third handle: one mixed backward equals the mix of the two
    gh = G.GpuBom(wl, p_in, out_mode=B.BOM_OUT_G_AND_H)
    gh.q.copy_(fz.q)
    o2 = gh.step(x, y, t_chk)
    for k, u in enumerate(gout["grads"]):
        mix = (1 - LAM) * o2["grads"][k].double() + LAM * o2["h"][k].double()
        assert G.rel_l2(G.np64(u), G.np64(mix)) < TOL, k
    del o2, gh, gout, us
    torch.cuda.empty_cache()

    # the fused step the bench times
    fz.model.step(xd, yd, wl.n_rows, fz.params, fz.q, t_chk, None, None)
    assert fz.model.stats()["code"] == B.BOM_OK
    th_out = [_dev_rows(a, r) for a, r in zip(theta, rows)]
    v_out = [_dev_rows(a, r) for a, r in zip(v, rows)]

    # the oracle on the same inputs
    p64 = [G.np64(p) for p in p_in]
    del p_in
    layers = X.oracle_layers(wl)
    Z, saved = O.forward(layers, False, p64, I.bf16_to_f64(x))
    ref = _task_space(Z, y, q_in.astype(np.float32), t_chk)
    del Z
    _check_task_space({"stats": fz.model.stats(), "q": G.np64(fz.q), **_outputs(fz.model, wl)}, ref)
    want = O.mix_grad_rows(layers, False, p64, saved, ref["R"], ref["valid"], ref["qhat"], ref["n_t"], LAM, rows)
    del saved, ref
    worst = {}
    for k in range(len(params)):
        e_u = G.rel_l2(u_rows[k], want[k])
        th_ref, v_ref = O.bom_update(th_in[k], want[k], v_in[k], F(lr), F(wds[k]), t_chk, F(b2), F(eps))
        e_th = G.rel_l2(th_out[k], th_ref)
        e_v = G.rel_l2(v_out[k], v_ref)
        e_step, bound = G.weighted_step_check(th_out[k], th_in[k], th_ref, v_ref, t_chk, b2, TOL)
        worst[k] = (e_u, e_th, e_v, e_step / bound)
        assert e_u < TOL, (k, e_u)
        assert e_th < TOL and e_v < TOL and e_step <= bound, (k, e_th, e_v, e_step, bound)
    print("LM block full size, rel L2 per tensor (u, theta, v; weighted step / its bound):",
          {k: tuple(f"{e:.2e}" for e in w) for k, w in worst.items()})


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
