"""Checkpoint and resume, and non-finite logits.

BOM's whole optimizer state is theta (the fp32 master weights), v, q and t:
about 8 bytes per parameter against AdamW's 12 (the cost-accounting appendix),
because the first moment lives in the d_out-sized q.  A run that saves that
state to the host after k steps, tears down its buffers and handle, restores
the state into fresh ones and continues must match an uninterrupted run to the
bit: every reduction of the step has a fixed order, and the compute copy of a
weight is the rounded master.

A step whose logits are not finite latches BOM_ENONFINITE before anything
writes q, theta, v, the compute copy or the device step counter."""
import numpy as np
import pytest
import torch

from paper_2609_36738_gb300 import bom as B
from paper_2609_36738_gb300 import inputs as I
from tests import _gpu as G

pytestmark = pytest.mark.gpu
LR, B2, EPS, WD = 1e-3, 0.999, 1e-8, 0.01


@pytest.fixture(scope="module", autouse=True)
def _built():
    G.ensure_built()


class Trainer:
    """A handle with the fused update, built from a saved state or from the
    workload's initial parameters."""

    def __init__(self, wl, seed, state=None, device_t=False):
        self.wl, self.seed = wl, seed
        bf16 = wl.dtype == "bf16"
        if state is None:
            init = I.init_params(wl, seed)
            theta = [I.bf16_to_f32(p) if bf16 else p.copy() for p in init]
            v = [np.zeros(a.shape, dtype=np.float32) for a in theta]
            q = np.zeros(wl.vocab, dtype=np.float32)
            t = 1
        else:
            theta, v, q, t = state["theta"], state["v"], state["q"], state["t"]
        self.theta = [torch.from_numpy(np.ascontiguousarray(a)).to(G.DEV) for a in theta]
        self.v = [torch.from_numpy(np.ascontiguousarray(a)).to(G.DEV) for a in v]
        self.q = torch.from_numpy(np.ascontiguousarray(q)).to(G.DEV)
        # the compute copy is the master rounded to the compute dtype
        self.params = [a.to(torch.bfloat16) if bf16 else a.clone() for a in self.theta]
        self.t = t
        self.model = B.BomModel(B.config_for(wl))
        B.bom_set_fused_update(self.model.h, self.theta, self.v, I.weight_decay_mask(wl, WD), LR, B2, EPS)
        self.t_dev = None
        if device_t:
            self.t_dev = torch.full((1,), t, dtype=torch.int64, device=G.DEV)
            B.bom_set_step_scalars(self.model.h, self.t_dev, None)

    def step(self, x=None, check=True):
        if x is None:
            x, y = I.make_batch(self.wl, self.seed, self.t)
        else:
            _, y = I.make_batch(self.wl, self.seed, self.t)
        xd = G.to_dev(x)
        yd = torch.from_numpy(np.ascontiguousarray(y, dtype=np.int32)).to(G.DEV)
        self.model.step(xd, yd, xd.shape[0], self.params, self.q, 0 if self.t_dev is not None else self.t, None,
                        None)
        st = self.model.stats(check=check)
        if st["code"] == B.BOM_OK:
            self.t += 1
        return st

    def save(self):
        torch.cuda.synchronize()
        t = int(self.t_dev.item()) if self.t_dev is not None else self.t
        return {"theta": [a.cpu().numpy() for a in self.theta], "v": [a.cpu().numpy() for a in self.v],
                "q": self.q.cpu().numpy(), "t": t}

    def state(self):
        return [self.q] + self.theta + self.v + self.params

    def close(self):
        self.model.close()


@pytest.mark.parametrize("name", ["tiny_mlp_f32", "tiny_norm_f32", "vision_small", "lm_mlp_small"])
@pytest.mark.parametrize("device_t", [False, True])
def test_resume_from_checkpoint_is_bit_equal(name, device_t):
    wl = I.WORKLOADS[name]
    straight = Trainer(wl, 21, device_t=device_t)
    for _ in range(6):
        straight.step()
    first = Trainer(wl, 21, device_t=device_t)
    for _ in range(3):
        first.step()
    ck = first.save()
    first.close()
    del first
    # the saved state is theta and v (8 bytes per parameter), q and t
    P = sum(a.size for a in ck["theta"])
    assert sum(a.nbytes for a in ck["theta"] + ck["v"]) == 8 * P
    assert ck["q"].nbytes == 4 * wl.vocab and ck["t"] == 4
    resumed = Trainer(wl, 21, state=ck, device_t=device_t)
    for _ in range(3):
        resumed.step()
    torch.cuda.synchronize()
    for k, (a, b) in enumerate(zip(straight.state(), resumed.state())):
        assert torch.equal(a, b), k
    if device_t:
        assert int(straight.t_dev.item()) == int(resumed.t_dev.item()) == 7


@pytest.mark.parametrize("name,bad", [("tiny_mlp_f32", float("nan")), ("lm_mlp_small", float("inf")),
                                      ("vision_small", float("nan"))])
def test_nonfinite_logits_leave_state_unchanged(name, bad):
    wl = I.WORKLOADS[name]
    tr = Trainer(wl, 22, device_t=True)
    tr.step()
    torch.cuda.synchronize()
    before = [a.clone() for a in tr.state()]
    x, _ = I.make_batch(wl, 22, tr.t)
    x = x.copy()
    if x.dtype == np.uint16:
        x[wl.n_rows // 3, 1] = I.bf16_bits(np.array([bad], dtype=np.float32))[0]
    else:
        x[wl.n_rows // 3, 1] = bad
    st = tr.step(x, check=False)
    assert st["code"] == B.BOM_ENONFINITE
    torch.cuda.synchronize()
    assert int(tr.t_dev.item()) == 2
    for a, b in zip(before, tr.state()):
        assert torch.equal(a, b)
    # the next finite step runs normally
    assert tr.step()["code"] == B.BOM_OK
    assert int(tr.t_dev.item()) == 3
