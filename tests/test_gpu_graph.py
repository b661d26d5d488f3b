"""Step scalars on the device and captured steps (bom_set_step_scalars,
bom_graph_capture / bom_graph_launch).

Algorithm 1 changes two scalars every step: the bias corrections
1/(1 - beta1^t) of q (Section 3.2) and 1/(1 - beta2^t) of v (Section 3.4),
and usually the learning rate.  With a device step counter a step reads them
from device memory, so one captured step can be replayed for every later
step.  Replayed and directly launched steps must agree to the bit: the same
kernels run on the same inputs, and the corrections the device forms from t
equal the ones the host forms."""
import numpy as np
import pytest
import torch

from paper_2609_36738_gb300 import bom as B
from paper_2609_36738_gb300 import inputs as I
from tests import _gpu as G

pytestmark = pytest.mark.gpu
LR, B2, EPS, WD = 1e-3, 0.999, 1e-8, 0.01
NAMES = ["tiny_mlp_f32", "tiny_norm_f32", "vision_small", "lm_head_small", "lm_mlp_small", "lm_norm_small"]


@pytest.fixture(scope="module", autouse=True)
def _built():
    G.ensure_built()


class Run:
    """A handle with the fused update registered and resident input buffers."""

    def __init__(self, wl, seed, device_scalars):
        self.wl = wl
        params = I.init_params(wl, seed)
        self.gpu = G.GpuBom(wl, params)
        self.theta = [torch.from_numpy(I.bf16_to_f32(p) if wl.dtype == "bf16" else p.copy()).to(G.DEV)
                      for p in params]
        self.v = [torch.zeros(p.shape, dtype=torch.float32, device=G.DEV) for p in params]
        self.wd = I.weight_decay_mask(wl, WD)
        B.bom_set_fused_update(self.gpu.model.h, self.theta, self.v, self.wd, LR, B2, EPS)
        x, y = I.make_batch(wl, seed, 1)
        self.x = G.to_dev(x)
        self.y = torch.from_numpy(np.ascontiguousarray(y, dtype=np.int32)).to(G.DEV)
        self.t_dev = self.lr_dev = None
        if device_scalars:
            self.t_dev = torch.ones(1, dtype=torch.int64, device=G.DEV)
            self.lr_dev = torch.full((1,), LR, dtype=torch.float32, device=G.DEV)
            B.bom_set_step_scalars(self.gpu.model.h, self.t_dev, self.lr_dev)

    def load(self, x, y):
        self.x.copy_(G.to_dev(x))
        self.y.copy_(torch.from_numpy(np.ascontiguousarray(y, dtype=np.int32)).to(G.DEV))

    def step(self, t):
        self.gpu.model.step(self.x, self.y, self.x.shape[0], self.gpu.params, self.gpu.q, t, None, None)

    def capture(self):
        return B.bom_graph_capture(self.gpu.model.h, self.x, self.y, self.x.shape[0], self.gpu.params, self.gpu.q,
                                   None, None)

    def state(self):
        return [self.gpu.q] + self.theta + self.v + self.gpu.params


def _assert_same(a, b, what):
    for k, (u, w) in enumerate(zip(a.state(), b.state())):
        assert torch.equal(u, w), (what, k)


@pytest.mark.parametrize("name", NAMES)
def test_device_step_scalars_equal_host_scalars(name):
    wl = I.WORKLOADS[name]
    host, dev = Run(wl, 11, False), Run(wl, 11, True)
    for t in range(1, 5):
        x, y = I.make_batch(wl, 11, t)
        host.load(x, y)
        dev.load(x, y)
        host.step(t)
        dev.step(0)   # t comes from the device counter
        st_h, st_d = host.gpu.model.stats(), dev.gpu.model.stats()
        assert st_h["loss"] == st_d["loss"] and st_h["n_t"] == st_d["n_t"]
        _assert_same(host, dev, t)
        assert int(dev.t_dev.item()) == t + 1


@pytest.mark.parametrize("name", NAMES)
def test_graph_replay_equals_direct_steps(name):
    wl = I.WORKLOADS[name]
    direct, graph = Run(wl, 12, False), Run(wl, 12, True)
    g = graph.capture()
    try:
        torch.cuda.synchronize()
        # capturing runs nothing
        assert int(graph.t_dev.item()) == 1
        assert not graph.gpu.q.any()
        lr = LR
        for t in range(1, 6):
            if t == 4:   # a new learning rate reaches the replay through lr_dev
                lr = LR / 2
                B.bom_set_fused_update(direct.gpu.model.h, direct.theta, direct.v, direct.wd, lr, B2, EPS)
                graph.lr_dev.fill_(lr)
            x, y = I.make_batch(wl, 12, t)
            direct.load(x, y)
            graph.load(x, y)
            direct.step(t)
            n0 = B.bom_launch_count()
            B.bom_graph_launch(g)
            assert B.bom_launch_count() > n0
            st_d, st_g = direct.gpu.model.stats(), graph.gpu.model.stats()
            assert st_d["loss"] == st_g["loss"] and st_d["n_t"] == st_g["n_t"]
            _assert_same(direct, graph, t)
            assert int(graph.t_dev.item()) == t + 1
    finally:
        B.bom_graph_destroy(g)


@pytest.mark.parametrize("name", ["lm_mlp_small", "tiny_mlp_f32", "vision_small"])
def test_device_counter_errors_leave_state_and_counter_unchanged(name):
    wl = I.WORKLOADS[name]
    r = Run(wl, 13, True)
    x, y = I.make_batch(wl, 13, 1)
    r.load(x, y)
    r.step(0)
    r.gpu.model.stats()
    before = [a.clone() for a in r.state()]
    # a counter below 1
    r.t_dev.fill_(0)
    r.step(0)
    st = r.gpu.model.stats(check=False)
    assert st["code"] == B.BOM_EINVAL
    assert int(r.t_dev.item()) == 0
    for a, b in zip(before, r.state()):
        assert torch.equal(a, b)
    # a label outside the vocabulary, replayed from a graph
    r.t_dev.fill_(2)
    g = r.capture()
    try:
        bad = y.copy()
        bad[5] = wl.vocab
        r.load(x, bad)
        B.bom_graph_launch(g)
        st = r.gpu.model.stats(check=False)
        assert st["code"] == B.BOM_ELABEL
        assert int(r.t_dev.item()) == 2
        for a, b in zip(before, r.state()):
            assert torch.equal(a, b)
        # the same graph runs the next valid step
        r.load(x, y)
        B.bom_graph_launch(g)
        assert r.gpu.model.stats()["code"] == B.BOM_OK
        assert int(r.t_dev.item()) == 3
    finally:
        B.bom_graph_destroy(g)


def test_graph_argument_checks():
    wl = I.TINY_MLP_F32
    r = Run(wl, 14, False)
    # no device step counter: a replay would repeat one t
    with pytest.raises(B.BomError) as e:
        r.capture()
    assert e.value.code == B.BOM_EINVAL
    # misaligned counters are refused on the host (the pointers are not dereferenced)
    base = torch.zeros(4, dtype=torch.int64, device=G.DEV)
    with pytest.raises(B.BomError) as e:
        B.bom_set_step_scalars(r.gpu.model.h, base.data_ptr() + 4, None)
    assert e.value.code == B.BOM_ENOTSUP
    with pytest.raises(B.BomError) as e:
        B.bom_set_step_scalars(r.gpu.model.h, base.data_ptr(), base.data_ptr() + 2)
    assert e.value.code == B.BOM_ENOTSUP
    # a bad step argument fails the capture and leaves no graph behind
    B.bom_set_step_scalars(r.gpu.model.h, base, None)
    with pytest.raises(B.BomError) as e:
        B.bom_graph_capture(r.gpu.model.h, r.x, r.y, wl.n_rows + 10**6, r.gpu.params, r.gpu.q, None, None)
    assert e.value.code == B.BOM_EINVAL
    B.bom_set_step_scalars(r.gpu.model.h, None, None)
    # a direct step still works after the failed capture
    r.step(1)
    assert r.gpu.model.stats()["code"] == B.BOM_OK
