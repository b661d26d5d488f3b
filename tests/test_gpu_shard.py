"""Row-sharded step: the data-parallel split of bom_step at its one exchange
(Algorithm 1: s_t and the surrogate use the mean over the supervised set I_t
of the whole batch; LM construction appendix: ignored targets leave both
means).  A batch is split by rows over two or three handles on one GPU; each
shard runs bom_step_shard_begin, the shards' exchange vectors are summed,
each shard runs bom_step_shard_end, and the shards' gradient shares are
added.  The result must equal the fp64 oracle's step of the whole batch:
N_t exactly, s_t, q_t, qhat_t, CE and u (or g and h) within the tolerance of
the path."""
import numpy as np
import pytest
import torch

from paper_2609_36738_gb300 import bom as B
from paper_2609_36738_gb300 import inputs as I
from tests import _gpu as G

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    G.ensure_built()


def _q0(V, seed=11):
    rng = np.random.default_rng(seed)
    q = (rng.standard_normal(V) * 0.01).astype(np.float32)
    return q - q.mean(dtype=np.float64).astype(np.float32)


def _run_shards(wl, params, x, y, q0, t, cuts, out_mode=B.BOM_OUT_U, check=True):
    """Both halves on every shard; returns the summed gradient shares (fp64
    host), per-shard results and the summed exchange vector."""
    V = wl.vocab
    bounds = [0, *cuts, wl.n_rows]
    shards = []
    for a, b in zip(bounds[:-1], bounds[1:]):
        g = G.GpuBom(wl, params, out_mode=out_mode, max_rows=b - a)
        g.q.copy_(torch.from_numpy(q0))
        xs = G.to_dev(np.ascontiguousarray(x[a:b]))
        ys = torch.from_numpy(np.ascontiguousarray(y[a:b], dtype=np.int32)).to(G.DEV)
        xch = torch.full((V + 3,), float("nan"), dtype=torch.float64, device=G.DEV)
        B.bom_step_shard_begin(g.model.h, xs, ys, b - a, g.params, xch)
        shards.append((g, xs, ys, b - a, xch))
    total = torch.zeros(V + 3, dtype=torch.float64, device=G.DEV)
    for *_, xch in shards:
        total += xch
    outs = []
    for g, xs, ys, n, _ in shards:
        grads = [torch.empty_like(p) for p in g.params]
        hs = ([torch.empty(p.shape, dtype=torch.float32, device=G.DEV) for p in g.params]
              if out_mode == B.BOM_OUT_G_AND_H else None)
        B.bom_step_shard_end(g.model.h, xs, ys, n, g.params, g.q, t, total, grads, hs)
        st = g.model.stats(check=check)
        o = dict(stats=st, grads=grads, h=hs, q=G.np64(g.q))
        if st["code"] == B.BOM_OK:
            qp, sp, _ = g.model.outputs()
            o["qhat"] = G.host_f32(qp, V)
            o["s"] = G.host_f32(sp, V)
        outs.append(o)
    return outs, G.np64(total)


def _sum(outs, key):
    return [sum(G.np64(o[key][k]) for o in outs) for k in range(len(outs[0][key]))]


CASES = [
    ("lm_mlp_mid", [137]),            # SwiGLU block, grouped weight gradients, ragged shards
    ("lm_mlp_mid", [64, 201]),        # three shards
    ("vision_small", [33]),           # Linear+GELU layers with biases, head bias
    ("lm_norm_small", [130]),         # RMSNorm before the head
    ("lm_head_small", [1]),           # a one-row shard
    ("tiny_ragged_f32", [20]),        # fp32 path
    ("tiny_norm_f32", [12, 24]),      # fp32 path with RMSNorm, three shards
]


@pytest.mark.parametrize("name, cuts", CASES)
def test_sharded_step_equals_the_whole_batch(name, cuts):
    wl = I.WORKLOADS[name]
    tol = G.TOL[wl.dtype]
    params = I.init_params(wl, 21)
    x, y = I.make_batch(wl, 21, 2)
    q0, t = _q0(wl.vocab), 3
    outs, total = _run_shards(wl, params, x, y, q0, t, cuts)
    ref = G.oracle_step(wl, X_params(wl, params), x, y, q0.astype(np.float64), t)
    assert total[wl.vocab + 1] == ref["n_t"] and total[wl.vocab + 2] == 0
    for o in outs:
        assert o["stats"]["n_t"] == ref["n_t"]
        assert abs(o["stats"]["loss"] - ref["ce"]) <= tol * abs(ref["ce"])
        for k in ("q", "qhat", "s"):
            assert G.rel_l2(o[k], ref[k]) < tol, k
        assert np.array_equal(o["q"], outs[0]["q"])   # every shard holds the same q
    u = _sum(outs, "grads")
    for k in range(len(u)):
        assert G.rel_l2(u[k], ref["u"][k]) < tol, (name, k, G.rel_l2(u[k], ref["u"][k]))


@pytest.mark.parametrize("name, cuts", [("lm_mlp_mid", [150]), ("vision_small", [40]), ("tiny_ragged_f32", [16])])
def test_sharded_step_g_and_h(name, cuts):
    wl = I.WORKLOADS[name]
    tol = G.TOL[wl.dtype]
    params = I.init_params(wl, 22)
    x, y = I.make_batch(wl, 22, 1)
    q0, t = _q0(wl.vocab, 12), 2
    outs, _ = _run_shards(wl, params, x, y, q0, t, cuts, out_mode=B.BOM_OUT_G_AND_H)
    ref = G.oracle_step(wl, X_params(wl, params), x, y, q0.astype(np.float64), t)
    g, h = _sum(outs, "grads"), _sum(outs, "h")
    for k in range(len(g)):
        assert G.rel_l2(g[k], ref["g"][k]) < tol, k
        assert G.rel_l2(h[k], ref["h"][k]) < tol, k


def test_a_shard_without_supervised_rows():
    """A shard whose rows are all ignored contributes its activations' nothing
    to s_t and N_t, and the step still equals the whole batch's."""
    wl = I.LM_MLP_MID
    params = I.init_params(wl, 23)
    x, y = I.make_batch(wl, 23, 1)
    y = y.copy()
    y[:90] = I.IGNORE_INDEX
    q0 = _q0(wl.vocab, 13)
    outs, total = _run_shards(wl, params, x, y, q0, 4, [90])
    ref = G.oracle_step(wl, X_params(wl, params), x, y, q0.astype(np.float64), 4)
    assert total[wl.vocab + 1] == ref["n_t"]
    u = _sum(outs, "grads")
    for k in range(len(u)):
        assert G.rel_l2(u[k], ref["u"][k]) < G.TOL["bf16"], k
    assert outs[0]["stats"]["n_t"] == ref["n_t"]


def test_errors_stop_every_shard_and_leave_q():
    wl = I.LM_MLP_MID
    params = I.init_params(wl, 24)
    x, y = I.make_batch(wl, 24, 1)
    q0 = _q0(wl.vocab, 14)
    # a bad label in the second shard: that shard latches BOM_ELABEL, the
    # first one BOM_ESHARD through the summed flag; q stays as it was
    yb = y.copy()
    yb[250] = wl.vocab
    outs, total = _run_shards(wl, params, x, yb, q0, 2, [150], check=False)
    assert total[wl.vocab + 2] == 1
    assert outs[0]["stats"]["code"] == B.BOM_ESHARD
    assert outs[1]["stats"]["code"] == B.BOM_ELABEL
    for o in outs:
        assert np.array_equal(o["q"], q0.astype(np.float64))
    # no supervised row in the whole batch: every shard latches BOM_EEMPTY
    ye = np.full_like(y, I.IGNORE_INDEX)
    outs, total = _run_shards(wl, params, x, ye, q0, 2, [150], check=False)
    assert total[wl.vocab + 1] == 0
    for o in outs:
        assert o["stats"]["code"] == B.BOM_EEMPTY
        assert np.array_equal(o["q"], q0.astype(np.float64))


def test_host_checks_of_the_sharded_calls():
    wl = I.LM_HEAD_SMALL
    g = G.GpuBom(wl, I.init_params(wl, 0))
    x, y = I.make_batch(wl, 0, 1)
    xd, yd = G.to_dev(x), torch.from_numpy(y).to(G.DEV)
    xch = torch.zeros(wl.vocab + 3, dtype=torch.float64, device=G.DEV)
    grads = [torch.empty_like(p) for p in g.params]
    # a second half without its first half
    with pytest.raises(B.BomError) as e:
        B.bom_step_shard_end(g.model.h, xd, yd, wl.n_rows, g.params, g.q, 1, xch, grads)
    assert e.value.code == B.BOM_EINVAL
    # a misaligned exchange vector
    with pytest.raises(B.BomError) as e:
        B.bom_step_shard_begin(g.model.h, xd, yd, wl.n_rows, g.params, xch.data_ptr() + 4)
    assert e.value.code == B.BOM_ENOTSUP
    # a first half of a different size than the second
    B.bom_step_shard_begin(g.model.h, xd, yd, wl.n_rows, g.params, xch)
    with pytest.raises(B.BomError) as e:
        B.bom_step_shard_end(g.model.h, xd, yd, wl.n_rows - 1, g.params, g.q, 1, xch, grads)
    assert e.value.code == B.BOM_EINVAL
    # not with the fused update registered
    th = [torch.zeros(p.shape, dtype=torch.float32, device=G.DEV) for p in g.params]
    vv = [torch.zeros_like(a) for a in th]
    B.bom_set_fused_update(g.model.h, th, vv, [0.0] * len(th), 1e-3, 0.999, 1e-8)
    with pytest.raises(B.BomError) as e:
        B.bom_step_shard_begin(g.model.h, xd, yd, wl.n_rows, g.params, xch)
    assert e.value.code == B.BOM_EINVAL
    torch.cuda.synchronize()


def X_params(wl, params):
    from tests import _indep as X
    return X.params_f64(wl, params)
