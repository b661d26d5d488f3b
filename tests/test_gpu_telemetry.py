"""Drift telemetry and the own-step control on the GPU, through the C ABI,
against the fp64 oracle (Section 3.3, Eq. drift-telemetry; stale-control and
drift-measurement appendices).

Each step runs in BOM_OUT_G_AND_H mode with an own-step output registered, so
one bom_step yields g, h = Jbar^T qhat and o = Jbar^T s_t; bom_own_step_moment
then forms M_t, Mhat_t and the drift sums per group (head / encoder), and the
own-step control updates with u = (1 - lambda) g + lambda Mhat.  Every step is
compared with the oracle on the inputs the GPU step read (its parameters,
q_{t-1} and M_{t-1})."""
import math

import numpy as np
import pytest
import torch

import oracle as O
from paper_2609_36738_gb300 import bom as B
from paper_2609_36738_gb300 import inputs as I
from tests import _gpu as G
from tests import _indep as X

pytestmark = pytest.mark.gpu
LAM, B1, B2, EPS, LR = 0.5, 0.9, 0.999, 1e-8, 1e-3


@pytest.fixture(scope="module", autouse=True)
def _built():
    G.ensure_built()


def _groups(wl):
    """Tensor indices of the classification head and of the encoder (the rest)."""
    n = len(wl.param_shapes())
    nh = 2 if wl.head_bias else 1
    return list(range(n - nh, n)), list(range(n - nh))


@pytest.mark.parametrize("name", ["tiny_mlp_f32", "tiny_ragged_f32", "vision_small", "lm_head_small",
                                  "lm_mlp_small", "lm_norm_small"])
def test_own_step_control_with_drift_telemetry(name):
    wl = I.WORKLOADS[name]
    tol = G.TOL[wl.dtype]
    steps = 4
    params = I.init_params(wl, seed=9)
    gpu = G.GpuBom(wl, params, out_mode=B.BOM_OUT_G_AND_H)
    dev = G.DEV
    f32 = torch.float32
    o_buf = [torch.empty(p.shape, dtype=f32, device=dev) for p in gpu.params]
    B.bom_set_own_step_output(gpu.model.h, o_buf)
    M = [torch.zeros(p.shape, dtype=f32, device=dev) for p in gpu.params]
    mhat = [torch.zeros(p.shape, dtype=f32, device=dev) for p in gpu.params]
    master = [torch.from_numpy(I.bf16_to_f32(p) if wl.dtype == "bf16" else p).to(dev) for p in params]
    vs = [torch.zeros(p.shape, dtype=f32, device=dev) for p in params]
    wds = I.weight_decay_mask(wl, 0.01)
    F = lambda v: float(np.float32(v))
    head, enc = _groups(wl)
    layers = X.oracle_layers(wl)
    for t in range(1, steps + 1):
        x, y = I.make_batch(wl, seed=9, step=t)
        p_in = [G.np64(p) for p in gpu.params]
        q_in = G.np64(gpu.q)
        M_in = [G.np64(m) for m in M]
        th_in = [G.np64(m) for m in master]
        v_in = [G.np64(v) for v in vs]
        gout = gpu.step(x, y, t)
        ref = G.oracle_step(wl, p_in, x, y, q_in, t, lam=LAM, beta1=B1)
        o_ref, s_ref, n_t = O.own_step_projection(layers, wl.head_bias, p_in, X.x_f64(wl, x), y)
        assert gout["stats"]["n_t"] == n_t == ref["n_t"]
        for k in range(len(params)):
            assert G.rel_l2(G.np64(o_buf[k]), o_ref[k]) < tol, ("o", t, k)
        # within-batch cancellation
        ratio, s_norm, mean_norm = O.cancellation_ratio(ref["R"], ref["valid"], n_t)
        st = gout["stats"]
        assert abs(st["r_norm_mean"] - mean_norm) <= tol * mean_norm
        assert abs(st["cancel"] - ratio) <= 2 * tol * ratio
        # moment, Mhat and the drift sums of each group
        sums = {g: torch.zeros(4, dtype=torch.float64, device=dev) for g in ("head", "enc")}
        mh_ref = []
        for k in range(len(params)):
            grp = "head" if k in head else "enc"
            B.bom_own_step_moment(gpu.model.h, M[k], o_buf[k], gout["h"][k], mhat[k], M[k].numel(), B1, t,
                                  sums[grp])
            _, mr = O.own_step_moment(M_in[k], o_ref[k], t, B1)
            mh_ref.append(mr)
        torch.cuda.synchronize()
        for k in range(len(params)):
            assert G.rel_l2(G.np64(mhat[k]), mh_ref[k]) < tol, ("mhat", t, k)
        if wl.head_bias:   # Jbar_b = I: the bias moment is qhat itself
            assert G.rel_l2(G.np64(mhat[head[-1]]), gout["qhat"]) < 1e-5
        for grp, idx in (("head", head), ("enc", enc)):
            if not idx:
                continue
            a = np.concatenate([G.np64(mhat[k]).ravel() for k in idx])
            b = np.concatenate([G.np64(gout["h"][k]).ravel() for k in idx])
            exact = np.array([a @ b, a @ a, b @ b, (a - b) @ (a - b)])
            got = G.np64(sums[grp])
            assert np.all(np.abs(got - exact) <= 1e-5 * np.abs(exact) + 1e-30), (grp, got, exact)
            cos = got[0] / math.sqrt(got[1] * got[2])
            rel = math.sqrt(got[3] / got[1])
            sr = O.drift_statistics([mh_ref[k] for k in idx], [ref["h"][k] for k in idx])
            assert abs(cos - sr["cos"]) <= 3 * tol, (grp, t, cos, sr["cos"])
            if t == 1:      # qhat_1 = s_1: no drift yet
                assert rel <= tol
            else:
                assert abs(rel - sr["rel"]) <= 3 * tol * max(1.0, sr["rel"]), (grp, t, rel, sr["rel"])
        # own-step control update: u = (1 - lambda) g + lambda Mhat
        for k in range(len(params)):
            gt = B.BOM_BF16 if wl.dtype == "bf16" else B.BOM_F32
            shadow = gpu.params[k] if wl.dtype == "bf16" else None
            B.bom_update(master[k], gout["grads"][k], gt, mhat[k], vs[k], shadow, master[k].numel(), LR, wds[k],
                         LAM, B2, EPS, t)
        torch.cuda.synchronize()
        for k in range(len(params)):
            if wl.dtype == "f32":
                gpu.params[k].copy_(master[k])
            # the update applied to the GPU's own g and Mhat: fp32 arithmetic
            # against fp64, so the steps agree to rounding
            u_gpu = O.mix_numerator(G.np64(gout["grads"][k]), G.np64(mhat[k]), F(LAM))
            th_exp, _ = O.bom_update(th_in[k], u_gpu, v_in[k], F(LR), F(wds[k]), t, F(B2), F(EPS))
            d_gpu, d_exp = G.np64(master[k]) - th_in[k], th_exp - th_in[k]
            ulp = np.spacing(np.abs(th_in[k]).astype(np.float32)).astype(np.float64)
            assert np.all(np.abs(d_gpu - d_exp) <= 2 * ulp + 1e-4 * np.abs(d_exp)), ("theta", t, k)
            # and the oracle's own-step control step from the same inputs
            u_ref = O.mix_numerator(ref["g"][k], mh_ref[k], F(LAM))
            th_ref, _ = O.bom_update(th_in[k], u_ref, v_in[k], F(LR), F(wds[k]), t, F(B2), F(EPS))
            assert G.rel_l2(G.np64(master[k]), th_ref) < tol, ("theta", t, k)
    B.bom_set_own_step_output(gpu.model.h, None)


def test_own_step_output_argument_checks():
    wl = I.TINY_MLP_F32
    gpu = G.GpuBom(wl, I.init_params(wl, seed=0))
    n = len(gpu.params)
    bufs = [torch.empty(p.shape, dtype=torch.float32, device=G.DEV) for p in gpu.params]
    with pytest.raises(B.BomError) as e:
        B.bom_set_own_step_output(gpu.model.h, bufs[:-1] + [0])
    assert e.value.code == B.BOM_EINVAL
    base = torch.empty(1024, dtype=torch.float32, device=G.DEV)
    with pytest.raises(B.BomError) as e:
        B.bom_set_own_step_output(gpu.model.h, bufs[:-1] + [base.data_ptr() + 4])
    assert e.value.code == B.BOM_ENOTSUP
    m = torch.zeros(8, dtype=torch.float32, device=G.DEV)
    with pytest.raises(B.BomError) as e:     # sums without h
        B.bom_own_step_moment(gpu.model.h, m, m, None, m, 8, 0.9, 1,
                              torch.zeros(4, dtype=torch.float64, device=G.DEV))
    assert e.value.code == B.BOM_EINVAL
    with pytest.raises(B.BomError) as e:
        B.bom_own_step_moment(gpu.model.h, m, m, m, m, 8, 0.9, 0)
    assert e.value.code == B.BOM_EINVAL
    assert n == 4
