"""The BOM-AdamW update fused into bom_step (bom_set_fused_update) against the
oracle's step and update on the same inputs (Section 3.4; Algorithm 1, last
two steps), and against the separate update kernel where both must agree to
the bit (fp32 workloads, whose u is not rounded in either path)."""
import numpy as np
import pytest
import torch

import oracle as O
from paper_2609_36738_gb300 import bom as B
from paper_2609_36738_gb300 import inputs as I
from tests import _gpu as G

pytestmark = pytest.mark.gpu
LR, B2, EPS, WD = 1e-3, 0.999, 1e-8, 0.01
F = lambda x: float(np.float32(x))


@pytest.fixture(scope="module", autouse=True)
def _built():
    G.ensure_built()


class Fused:
    """A handle with the fused update registered, its fp32 masters and v."""

    def __init__(self, wl, seed):
        self.wl = wl
        params = I.init_params(wl, seed)
        self.gpu = G.GpuBom(wl, params)
        self.theta = [torch.from_numpy(I.bf16_to_f32(p) if wl.dtype == "bf16" else p.copy()).to(G.DEV)
                      for p in params]
        self.v = [torch.zeros(p.shape, dtype=torch.float32, device=G.DEV) for p in params]
        self.wd = I.weight_decay_mask(wl, WD)
        B.bom_set_fused_update(self.gpu.model.h, self.theta, self.v, self.wd, LR, B2, EPS)

    def step(self, x, y, t, check=True):
        xd = G.to_dev(x)
        yd = torch.from_numpy(np.ascontiguousarray(y, dtype=np.int32)).to(G.DEV)
        self.gpu.model.step(xd, yd, xd.shape[0], self.gpu.params, self.gpu.q, t, None, None)
        return self.gpu.model.stats(check=check)


# Up to 1024 rows the bf16 step writes u and updates every tensor in one
# launch after the pass; lm_mlp_k1100 (1100 rows) takes the update in the
# weight-gradient GEMMs' epilogues, as the full-size LM block does.
# vision_mid and vision_head_bf16 (300 and 256 rows) take the bias gradients
# from the column sums of 32-row blocks formed in the cotangent GEMMs.
@pytest.mark.parametrize("name", ["tiny_mlp_f32", "tiny_ragged_f32", "tiny_norm_f32", "tiny_bf16", "vision_small",
                                  "vision_mid", "vision_head_bf16", "vision_wide", "lm_head_small", "lm_mlp_small",
                                  "lm_norm_small", "lm_head_wide", "lm_mlp_mid", "lm_mlp_k1100"])
def test_fused_update_matches_oracle_on_the_same_inputs(name):
    wl = I.WORKLOADS[name]
    tol = G.TOL[wl.dtype]
    f = Fused(wl, seed=3)
    for t in range(1, 5):
        x, y = I.make_batch(wl, seed=3, step=t)
        p_in = [G.np64(p) for p in f.gpu.params]
        q_in = G.np64(f.gpu.q)
        th_in = [G.np64(a) for a in f.theta]
        v_in = [G.np64(a) for a in f.v]
        st = f.step(x, y, t)
        torch.cuda.synchronize()
        ref = G.oracle_step(wl, p_in, x, y, q_in, t)
        assert st["n_t"] == ref["n_t"]
        assert G.rel_l2(G.np64(f.gpu.q), ref["q"]) < tol
        shapes = wl.param_shapes()
        for k in range(len(p_in)):
            th_ref, v_ref = O.bom_update(th_in[k], ref["u"][k], v_in[k], F(LR), F(f.wd[k]), t, F(B2), F(EPS))
            th = G.np64(f.theta[k])
            # the step, weighed by each element's own sqrt(vhat)
            err, bound = G.weighted_step_check(th, th_in[k], th_ref, v_ref, t, B2, tol)
            assert err <= bound, (t, k, err, bound)
            assert G.rel_l2(G.np64(f.v[k]), v_ref) < tol, (t, k)
            if shapes[k][2]:
                # weights start far from zero; a zero-initialised vector's
                # theta is a sum of steps of about lr each, checked above
                assert G.rel_l2(th, th_ref) < tol, (t, k)
            # the compute copy is the rounded master
            cp = f.theta[k].to(f.gpu.params[k].dtype).view(f.gpu.params[k].shape)
            assert torch.equal(f.gpu.params[k], cp), (t, k)


@pytest.mark.parametrize("name", ["tiny_mlp_f32", "tiny_norm_f32"])
def test_fused_equals_separate_update_bitwise_fp32(name):
    """fp32: the separate path stores u in fp32 and updates it with the same
    arithmetic, so theta, v and the parameters agree to the bit."""
    wl = I.WORKLOADS[name]
    f = Fused(wl, seed=4)
    sep = G.GpuBom(wl, I.init_params(wl, 4))
    th2 = [a.clone() for a in f.theta]
    v2 = [a.clone() for a in f.v]
    for t in range(1, 4):
        x, y = I.make_batch(wl, seed=4, step=t)
        f.step(x, y, t)
        out = sep.step(x, y, t)
        for k in range(len(th2)):
            B.bom_update(th2[k], out["grads"][k], B.BOM_F32, None, v2[k], None, th2[k].numel(), LR, f.wd[k], 0.5,
                         B2, EPS, t)
            sep.params[k].copy_(th2[k])
        torch.cuda.synchronize()
        for k in range(len(th2)):
            assert torch.equal(f.theta[k], th2[k]), (t, k)
            assert torch.equal(f.v[k], v2[k]), (t, k)
            assert torch.equal(f.gpu.params[k], sep.params[k]), (t, k)


def test_fused_update_is_deterministic_and_skips_failed_steps():
    wl = I.LM_MLP_SMALL
    runs = []
    for _ in range(2):
        f = Fused(wl, seed=5)
        for t in range(1, 4):
            x, y = I.make_batch(wl, seed=5, step=t)
            f.step(x, y, t)
        torch.cuda.synchronize()
        runs.append(f)
    for a, b in zip(runs[0].theta + runs[0].v + runs[0].gpu.params, runs[1].theta + runs[1].v + runs[1].gpu.params):
        assert torch.equal(a, b)
    # a step whose labels are invalid latches an error and leaves everything unchanged
    f = runs[0]
    before = [a.clone() for a in f.theta + f.v + f.gpu.params]
    x, y = I.make_batch(wl, seed=5, step=9)
    y = y.copy()
    y[3] = wl.vocab
    st = f.step(x, y, 4, check=False)
    assert st["code"] == B.BOM_ELABEL
    for a, b in zip(before, f.theta + f.v + f.gpu.params):
        assert torch.equal(a, b)


def test_fused_update_argument_checks():
    wl = I.TINY_MLP_F32
    f = Fused(wl, seed=0)
    x, y = I.make_batch(wl, seed=0, step=1)
    gh = G.GpuBom(wl, I.init_params(wl, 0), out_mode=B.BOM_OUT_G_AND_H)
    with pytest.raises(B.BomError) as e:      # the fused update needs the u pass
        B.bom_set_fused_update(gh.model.h, f.theta, f.v, f.wd, LR, B2, EPS)
        gh.step(x, y, 1)
    assert e.value.code == B.BOM_EINVAL
    with pytest.raises(B.BomError) as e:
        B.bom_set_fused_update(f.gpu.model.h, f.theta[:-1] + [0], f.v, f.wd, LR, B2, EPS)
    assert e.value.code == B.BOM_EINVAL
    B.bom_set_fused_update(f.gpu.model.h, None, None, None, 0.0, 0.0, 0.0)
    with pytest.raises(B.BomError):           # disabled again: grads are required
        f.step(x, y, 1)


def test_fused_update_on_rows_only_16_byte_aligned_gives_the_same_bits():
    """theta and v placed 16 bytes past a 32-byte boundary (the ABI asks for
    16-byte alignment only): the update epilogue takes its 128-bit form
    instead of its 256-bit one, with the same arithmetic per element, so
    theta, v and the compute copies equal those of an aligned run bit for
    bit.  lm_mlp_k1100 (1100 rows) applies the update in the weight-gradient
    GEMMs' epilogues."""
    wl = I.LM_MLP_K1100
    ref = Fused(wl, seed=6)
    off = Fused(wl, seed=6)

    def shifted(a):   # same values, data pointer 16 bytes past a 32-byte boundary
        buf = torch.zeros(a.numel() + 4, dtype=a.dtype, device=a.device)
        view = buf[4:].view(a.shape)
        view.copy_(a)
        assert view.data_ptr() % 32 == 16
        return view

    off.theta = [shifted(a) for a in off.theta]
    off.v = [shifted(a) for a in off.v]
    B.bom_set_fused_update(off.gpu.model.h, off.theta, off.v, off.wd, LR, B2, EPS)
    for t in range(1, 4):
        x, y = I.make_batch(wl, seed=6, step=t)
        ref.step(x, y, t)
        off.step(x, y, t)
    torch.cuda.synchronize()
    for a, b in zip(ref.theta + ref.v + ref.gpu.params, off.theta + off.v + off.gpu.params):
        assert torch.equal(a, b)
