"""bom_step (and bom_update in multi-step runs) against the fp64 oracle, element
by element, on the same seeded inputs.

Tolerances (relative L2): 1e-5 for the fp32 path, 2e-2 for bf16 paths; label
handling (N_t) bit-exact.  Workloads span several GEMM tiles with ragged
tails, ignored rows, every layer kind, and both output modes."""
import dataclasses

import numpy as np
import pytest
import torch

import oracle as O
from paper_2609_36738_gb300 import bom as B
from paper_2609_36738_gb300 import inputs as I
from tests import _gpu as G
from tests import _indep as X

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    G.ensure_built()


def _compare_step(wl, gout, oref, tol, check_g_h):
    st = gout["stats"]
    assert st["n_t"] == oref["n_t"]                                   # bit-exact count
    assert abs(st["loss"] - oref["ce"]) <= tol * abs(oref["ce"]) + 1e-6
    assert G.rel_l2(gout["s"], oref["s"]) < tol
    assert G.rel_l2(gout["q"], oref["q"]) < tol
    assert G.rel_l2(gout["qhat"], oref["qhat"]) < tol
    valid = oref["valid"]
    assert G.rel_l2(gout["lse"][valid], oref["lse"][valid]) < tol
    # zero-sum invariant of s (Section 3.1), at the kernel's precision
    assert abs(gout["s"].sum()) <= 1e-5 * np.abs(gout["s"]).sum() + 1e-7
    if check_g_h:
        for k, (g, ref) in enumerate(zip(gout["grads"], oref["g"])):
            assert G.rel_l2(G.np64(g), ref) < tol, f"g[{k}]"
        for k, (h, ref) in enumerate(zip(gout["h"], oref["h"])):
            assert G.rel_l2(G.np64(h), ref) < tol, f"h[{k}]"
    else:
        for k, (u, ref) in enumerate(zip(gout["grads"], oref["u"])):
            assert G.rel_l2(G.np64(u), ref) < tol, f"u[{k}] {G.rel_l2(G.np64(u), ref)}"


@pytest.mark.parametrize("name", ["tiny_mlp_f32", "tiny_ragged_f32", "tiny_norm_f32", "tiny_bf16", "lm_head_small",
                                  "lm_norm_small", "vision_small", "vision_wide",
                                  "lm_mlp_small", "lm_mlp_mid"])
@pytest.mark.parametrize("mode", [B.BOM_OUT_U, B.BOM_OUT_G_AND_H])
def test_single_step_parity(name, mode):
    wl = I.WORKLOADS[name]
    params = I.init_params(wl, seed=0)
    p64 = X.params_f64(wl, params)
    x, y = I.make_batch(wl, seed=0, step=1)
    gpu = G.GpuBom(wl, params, out_mode=mode)
    # a non-zero zero-sum history so that qhat and the bias correction matter
    rng = np.random.default_rng(1)
    q0 = (rng.standard_normal(wl.vocab) * 0.01).astype(np.float32)
    q0 -= q0.mean(dtype=np.float64).astype(np.float32)
    gpu.q.copy_(torch.from_numpy(q0))
    t = 3
    gout = gpu.step(x, y, t)
    oref = G.oracle_step(wl, p64, x, y, q0.astype(np.float64), t)
    _compare_step(wl, gout, oref, G.TOL[wl.dtype], mode == B.BOM_OUT_G_AND_H)


@pytest.mark.parametrize("name,steps", [("tiny_mlp_f32", 5), ("vision_small", 3), ("lm_mlp_small", 3),
                                        ("tiny_norm_f32", 3), ("lm_norm_small", 3)])
def test_multi_step_trajectory(name, steps):
    """Several BOM steps, each followed by the update of every tensor (fp32
    master parameters on the device, bf16 copies for the bf16 path).  Each
    step is checked on the inputs the GPU read, and the master weights against
    the oracle's own trajectory."""
    wl = I.WORKLOADS[name]
    lr, b2, eps, lam = 1e-3, 0.999, 1e-8, 0.5
    wds = I.weight_decay_mask(wl, 0.01)
    params = I.init_params(wl, seed=5)
    p64 = X.params_f64(wl, params)
    gpu = G.GpuBom(wl, params)
    master = [G.to_dev(p.astype(np.float64).astype(np.float32)) if wl.dtype == "f32" else
              torch.from_numpy(I.bf16_to_f32(p)).to(G.DEV) for p in params]
    vs = [torch.zeros(p.shape, dtype=torch.float32, device=G.DEV) for p in params]
    vo = [np.zeros(p.shape) for p in p64]
    q = np.zeros(wl.vocab)
    tol = G.TOL[wl.dtype]
    for t in range(1, steps + 1):
        x, y = I.make_batch(wl, seed=5, step=t)
        p_in = [G.np64(p) for p in gpu.params]
        q_in = G.np64(gpu.q)
        gout = gpu.step(x, y, t)
        # the step on the inputs the GPU read: its parameters and q_{t-1}
        _compare_step(wl, gout, G.oracle_step(wl, p_in, x, y, q_in, t), tol, False)
        # the oracle's own trajectory; bf16 workloads compute with bf16 copies
        # of the master weights on both sides
        pin = [G.bf16_round(p) for p in p64] if wl.dtype == "bf16" else p64
        oref = G.oracle_step(wl, pin, x, y, q, t)
        q = oref["q"]
        for k in range(len(params)):
            n = master[k].numel()
            gt = B.BOM_BF16 if wl.dtype == "bf16" else B.BOM_F32
            shadow = gpu.params[k] if wl.dtype == "bf16" else None
            B.bom_update(master[k], gout["grads"][k], gt, None, vs[k], shadow, n, lr, wds[k], lam, b2, eps, t)
            if wl.dtype == "f32":
                gpu.params[k].copy_(master[k])
            p64[k], vo[k] = O.bom_update(p64[k], oref["u"][k], vo[k], lr, wds[k], t, b2, eps)
        torch.cuda.synchronize()
        for k in range(len(params)):
            assert G.rel_l2(G.np64(master[k]), p64[k]) < tol


# lm_head_small: the cluster task pass; tiny_mlp_f32, tiny_bf16: the one-CTA
# shared-memory pass
@pytest.mark.parametrize("name", ["lm_head_small", "tiny_mlp_f32", "tiny_bf16"])
def test_device_errors_leave_q_unchanged(name):
    wl = I.WORKLOADS[name]
    params = I.init_params(wl, seed=0)
    x, y = I.make_batch(wl, seed=0, step=1)
    gpu = G.GpuBom(wl, params)
    gpu.q.fill_(0.25)
    bad = y.copy()
    bad[5] = wl.vocab
    out = gpu.step(x, bad, 1, check=False)
    assert out["stats"]["code"] == B.BOM_ELABEL
    assert torch.all(gpu.q == 0.25)
    out = gpu.step(x, np.full_like(y, I.IGNORE_INDEX), 1, check=False)
    assert out["stats"]["code"] == B.BOM_EEMPTY
    assert torch.all(gpu.q == 0.25)
    # the handle is usable again after an error
    out = gpu.step(x, y, 1)
    assert out["stats"]["code"] == B.BOM_OK


def test_host_checked_arguments():
    wl = I.LM_HEAD_SMALL
    params = I.init_params(wl, seed=0)
    x, y = I.make_batch(wl, seed=0, step=1)
    gpu = G.GpuBom(wl, params)
    xd = G.to_dev(x)
    yd = torch.from_numpy(y).to(G.DEV)
    grads = [torch.empty_like(p) for p in gpu.params]
    for kw in (dict(n=0, t=1), dict(n=wl.n_rows + 1, t=1), dict(n=wl.n_rows, t=0)):
        with pytest.raises(B.BomError) as e:
            gpu.model.step(xd, yd, kw["n"], gpu.params, gpu.q, kw["t"], grads)
        assert e.value.code == B.BOM_EINVAL


def test_deterministic_reruns():
    """Same inputs, same bits: every reduction of the step has a fixed order."""
    wl = I.LM_MLP_SMALL
    params = I.init_params(wl, seed=2)
    x, y = I.make_batch(wl, seed=2, step=1)
    a = G.GpuBom(wl, params).step(x, y, 1)
    b = G.GpuBom(wl, params).step(x, y, 1)
    assert np.array_equal(a["s"], b["s"]) and np.array_equal(a["q"], b["q"])
    for ga, gb in zip(a["grads"], b["grads"]):
        assert torch.equal(ga, gb)


@pytest.mark.parametrize("name", ["lm_head_small", "lm_mlp_small", "tiny_ragged_f32", "lm_head_wide",
                                  "tiny_norm_f32", "lm_norm_small"])
def test_input_cotangent(name):
    """bom_set_input_grad: the cotangent of X (for the head-only block this is
    dH, the input-side half of the head backward)."""
    wl = I.WORKLOADS[name]
    params = I.init_params(wl, seed=3)
    p64 = X.params_f64(wl, params)
    x, y = I.make_batch(wl, seed=3, step=1)
    gpu = G.GpuBom(wl, params)
    dx = torch.empty((wl.n_rows, wl.d_in), dtype=torch.bfloat16 if wl.dtype == "bf16" else torch.float32,
                     device=G.DEV)
    B.bom_set_input_grad(gpu.model.h, dx)
    gout = gpu.step(x, y, 1)
    oref = G.oracle_step(wl, p64, x, y, np.zeros(wl.vocab), 1)
    tol = G.TOL[wl.dtype]
    assert G.rel_l2(G.np64(dx), oref["dX_u"]) < tol
    for u, ref in zip(gout["grads"], oref["u"]):
        assert G.rel_l2(G.np64(u), ref) < tol


# A Qwen3-sized vocabulary on a small ragged batch: 151,936 columns give 1187
# column half-tiles per row to merge in the row log-sum-exp and a ragged last
# tile; the head's input-side GEMM contracts over all of them (split-K).
LM_HEAD_HUGE_V = dataclasses.replace(I.LM_HEAD_SMALL, name="lm_head_huge_vocab", n_rows=97, vocab=151_936)


@pytest.mark.parametrize("mode", [B.BOM_OUT_U, B.BOM_OUT_G_AND_H])
def test_huge_vocabulary_parity(mode):
    wl = LM_HEAD_HUGE_V
    params = I.init_params(wl, seed=2)
    p64 = X.params_f64(wl, params)
    x, y = I.make_batch(wl, seed=2, step=1)
    gpu = G.GpuBom(wl, params, out_mode=mode)
    gout = gpu.step(x, y, 1)
    oref = G.oracle_step(wl, p64, x, y, np.zeros(wl.vocab), 1)
    _compare_step(wl, gout, oref, G.TOL[wl.dtype], mode == B.BOM_OUT_G_AND_H)


@pytest.mark.parametrize("name", ["tiny_mlp_f32", "lm_mlp_small"])
def test_single_supervised_row(name):
    """N_t = 1: every label but one is the ignore index, so s_t is that row's
    residual and every mean is over one row."""
    wl = I.WORKLOADS[name]
    params = I.init_params(wl, seed=3)
    p64 = X.params_f64(wl, params)
    x, y = I.make_batch(wl, seed=3, step=1)
    y = np.full_like(y, I.IGNORE_INDEX)
    y[wl.n_rows // 2] = 5
    gpu = G.GpuBom(wl, params)
    gout = gpu.step(x, y, 2)
    oref = G.oracle_step(wl, p64, x, y, np.zeros(wl.vocab), 2)
    assert gout["stats"]["n_t"] == 1
    _compare_step(wl, gout, oref, G.TOL[wl.dtype], False)


def _guarded(shape, dtype, guard=64, fill=-7.25):
    """A tensor view of `shape` inside a buffer with `guard` sentinel elements
    on each side (16-byte aligned for both dtypes)."""
    n = int(np.prod(shape))
    buf = torch.full((guard + n + guard,), fill, dtype=dtype, device=G.DEV)
    return buf, buf[guard:guard + n].view(shape)


def _guards_intact(buf, n, guard=64, fill=-7.25):
    return bool((buf[:guard] == fill).all()) and bool((buf[guard + n:] == fill).all())


@pytest.mark.parametrize("name", ["tiny_ragged_f32", "tiny_norm_f32", "tiny_bf16", "vision_small", "lm_head_small",
                                  "lm_mlp_small", "lm_head_wide", "lm_norm_small"])
@pytest.mark.parametrize("mode", [B.BOM_OUT_U, B.BOM_OUT_G_AND_H])
def test_outputs_stay_inside_their_buffers(name, mode):
    """Canary regions around every output (u or g, h, the input cotangent and
    q): a step on ragged shapes writes none of them."""
    wl = I.WORKLOADS[name]
    params = I.init_params(wl, seed=4)
    x, y = I.make_batch(wl, seed=4, step=1)
    gpu = G.GpuBom(wl, params, out_mode=mode)
    cdt = torch.bfloat16 if wl.dtype == "bf16" else torch.float32
    gb = [_guarded(p.shape, cdt) for p in gpu.params]
    hb = [_guarded(p.shape, torch.float32) for p in gpu.params] if mode == B.BOM_OUT_G_AND_H else None
    dxb = _guarded((wl.n_rows, wl.d_in), cdt)
    qb = _guarded((wl.vocab,), torch.float32)
    qb[1].zero_()
    B.bom_set_input_grad(gpu.model.h, dxb[1])
    xd = G.to_dev(x)
    yd = torch.from_numpy(np.ascontiguousarray(y, dtype=np.int32)).to(G.DEV)
    gpu.model.step(xd, yd, wl.n_rows, gpu.params, qb[1], 1, [v for _, v in gb],
                   [v for _, v in hb] if hb else None)
    assert gpu.model.stats()["code"] == B.BOM_OK
    for buf, view in gb + (hb or []) + [dxb, qb]:
        assert _guards_intact(buf, view.numel())
        assert torch.isfinite(view.float()).all()
