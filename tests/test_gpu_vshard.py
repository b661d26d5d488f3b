"""Vocabulary-sharded step: the head's output columns split over two or three
handles on one GPU, every shard with the whole batch.  A row's residual
r_ij = exp(z_ij - lse_i) - [j = y_i] (Algorithm 1) needs the other columns only
through lse_i, s_t / q_t / qhat_t are per column (Section 3.2), and the head's
input cotangent a R W + b 1_{I_t} (W^T qhat)^T (Eq. mix-gradient) is a sum over
columns.  Each shard runs bom_step_vshard_begin; the test, as the caller,
stacks the shards' row log-sum-exp parts (the all-gather); each shard runs
bom_step_vshard_mid; the test sums their input-cotangent parts (the
all-reduce); each shard runs bom_step_vshard_end.  The result must equal the
fp64 oracle's step of the whole head: N_t exactly; the shards' q, qhat, s and
head rows of u, put side by side, the whole ones; every shard's backbone u the
whole batch's (and the same on every shard, bit for bit); the shards' CE parts
adding up to the loss."""
import dataclasses

import numpy as np
import pytest
import torch

from paper_2609_36738_gb300 import bom as B
from paper_2609_36738_gb300 import inputs as I
from tests import _gpu as G
from tests import _indep as X

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    G.ensure_built()


def _q0(V, seed=31):
    rng = np.random.default_rng(seed)
    q = (rng.standard_normal(V) * 0.01).astype(np.float32)
    return q - q.mean(dtype=np.float64).astype(np.float32)


def _head_index(wl):
    np_ = len(wl.param_shapes())
    return np_ - (2 if wl.head_bias else 1)


def _run_vshards(wl, params, x, y, q0, t, cuts, input_grad=False, check=True):
    """The three parts on every shard; returns per-shard results."""
    V, n, d = wl.vocab, wl.n_rows, wl.d_model
    hw = _head_index(wl)
    bounds = [0, *cuts, V]
    xd = G.to_dev(x)
    yd = torch.from_numpy(np.ascontiguousarray(y, dtype=np.int32)).to(G.DEV)
    shards = []
    for a, b in zip(bounds[:-1], bounds[1:]):
        wls = dataclasses.replace(wl, vocab=b - a)
        ps = list(params)
        ps[hw] = np.ascontiguousarray(params[hw][a:b])
        if wl.head_bias:
            ps[hw + 1] = np.ascontiguousarray(params[hw + 1][a:b])
        g = G.GpuBom(wls, ps)
        g.q.copy_(torch.from_numpy(q0[a:b]))
        dx = None
        if input_grad:
            dx = torch.full((n, wl.d_in), float("nan"), dtype=torch.bfloat16 if wl.dtype == "bf16" else torch.float32,
                            device=G.DEV)
            B.bom_set_input_grad(g.model.h, dx)
        part = torch.full((n,), float("nan"), dtype=torch.float32, device=G.DEV)
        B.bom_step_vshard_begin(g.model.h, xd, yd, n, g.params, V, a, part)
        shards.append(dict(g=g, a=a, b=b, part=part, dx=dx))
    parts = torch.stack([s["part"] for s in shards])   # the caller's all-gather, in shard order
    need_dh = len(wl.layers) > 0 or input_grad
    for s in shards:
        g = s["g"]
        s["grads"] = [torch.full_like(p, float("nan")) for p in g.params]
        s["dh"] = torch.full((n, d), float("nan"), dtype=torch.float32, device=G.DEV) if need_dh else None
        B.bom_step_vshard_mid(g.model.h, xd, yd, n, g.params, g.q, t, parts, len(shards), s["grads"], s["dh"])
        s["stats"] = g.model.stats(check=check)
        if s["stats"]["code"] == B.BOM_OK:
            qp, sp, lp = g.model.outputs()
            s["qhat"] = G.host_f32(qp, s["b"] - s["a"])
            s["s"] = G.host_f32(sp, s["b"] - s["a"])
            s["lse"] = G.host_f32(lp, n)
    dh_sum = None
    if need_dh:
        dh_sum = torch.zeros((n, d), dtype=torch.float32, device=G.DEV)
        for s in shards:   # the caller's all-reduce
            dh_sum += s["dh"]
    for s in shards:
        g = s["g"]
        B.bom_step_vshard_end(g.model.h, xd, yd, n, g.params, dh_sum, s["grads"])
        s["stats_end"] = g.model.stats(check=check)
        s["q"] = G.np64(g.q)
    return shards


def _compare(wl, shards, ref, tol, q0):
    hw = _head_index(wl)
    valid = ref["valid"]
    loss = 0.0
    for s in shards:
        assert s["stats"]["n_t"] == ref["n_t"]
        loss += s["stats"]["loss"]
        # every shard holds the same row log-sum-exp
        assert np.array_equal(s["lse"], shards[0]["lse"])
    assert abs(loss - ref["ce"]) <= tol * abs(ref["ce"])
    assert G.rel_l2(shards[0]["lse"][valid], ref["lse"][valid]) < tol
    for key in ("q", "qhat", "s"):
        got = np.concatenate([s[key] for s in shards])
        assert G.rel_l2(got, ref[key]) < tol, key
    u = ref["u"]
    # the head's rows: each shard's own, together the whole head
    head = np.concatenate([G.np64(s["grads"][hw]) for s in shards])
    assert G.rel_l2(head, u[hw]) < tol
    if wl.head_bias:
        hb = np.concatenate([G.np64(s["grads"][hw + 1]) for s in shards])
        assert G.rel_l2(hb, u[hw + 1]) < tol
    # the backbone: the whole batch's u on every shard, bit for bit the same
    for k in range(hw):
        for s in shards:
            assert torch.equal(s["grads"][k], shards[0]["grads"][k]), k
        assert G.rel_l2(G.np64(shards[0]["grads"][k]), u[k]) < tol, (k, G.rel_l2(G.np64(shards[0]["grads"][k]), u[k]))


CASES = [
    ("lm_mlp_mid", [500]),          # SwiGLU block: the backbone's backward runs from the summed cotangent
    ("lm_mlp_mid", [3, 700]),       # three shards, one of three columns
    ("vision_small", [64]),         # Linear+GELU layers (GELU' on the parts) and a head bias
    ("vision_wide", [250]),         # CTA-pair tiles in the backbone's backward
    ("lm_norm_small", [300]),       # RMSNorm before the head
    ("lm_head_wide", [4096]),       # split-K of the head's input-side GEMM on each shard
    ("tiny_ragged_f32", [3]),       # fp32 path
    ("tiny_norm_f32", [2, 5]),      # fp32 path with RMSNorm, three shards
]


@pytest.mark.parametrize("name, cuts", CASES)
def test_vocab_sharded_step_equals_the_whole_head(name, cuts):
    wl = I.WORKLOADS[name]
    tol = G.TOL[wl.dtype]
    params = I.init_params(wl, 41)
    x, y = I.make_batch(wl, 41, 2)
    q0, t = _q0(wl.vocab), 3
    shards = _run_vshards(wl, params, x, y, q0, t, cuts)
    ref = G.oracle_step(wl, X.params_f64(wl, params), x, y, q0.astype(np.float64), t)
    _compare(wl, shards, ref, tol, q0)
    for s in shards:
        assert s["stats_end"]["code"] == B.BOM_OK


def test_vocab_sharded_head_only_input_cotangent():
    """Head-only block with an input-gradient buffer: the last part writes the
    summed dH (the cotangent of the block's input) in the compute dtype."""
    wl = I.LM_HEAD_SMALL
    params = I.init_params(wl, 42)
    x, y = I.make_batch(wl, 42, 1)
    q0 = _q0(wl.vocab, 32)
    shards = _run_vshards(wl, params, x, y, q0, 2, [17, 600], input_grad=True)
    ref = G.oracle_step(wl, X.params_f64(wl, params), x, y, q0.astype(np.float64), 2)
    _compare(wl, shards, ref, G.TOL["bf16"], q0)
    for s in shards:
        assert torch.equal(s["dx"], shards[0]["dx"])
    assert G.rel_l2(G.np64(shards[0]["dx"]), ref["dX_u"]) < G.TOL["bf16"]


def test_device_step_counter_is_read_in_mid_and_advanced_in_end():
    wl = I.LM_MLP_MID
    params = I.init_params(wl, 43)
    x, y = I.make_batch(wl, 43, 1)
    q0 = _q0(wl.vocab, 33)
    t_devs = []
    orig = G.GpuBom.__init__

    def init(self, *a, **k):
        orig(self, *a, **k)
        td = torch.tensor([4], dtype=torch.int64, device=G.DEV)
        B.bom_set_step_scalars(self.model.h, td)
        t_devs.append(td)

    G.GpuBom.__init__ = init
    try:
        shards = _run_vshards(wl, params, x, y, q0, 1, [400])   # host t is ignored: t = 4 on the device
    finally:
        G.GpuBom.__init__ = orig
    ref = G.oracle_step(wl, X.params_f64(wl, params), x, y, q0.astype(np.float64), 4)
    _compare(wl, shards, ref, G.TOL["bf16"], q0)
    assert [int(td.item()) for td in t_devs] == [5, 5]


def test_errors_stop_every_shard_and_leave_q():
    wl = I.LM_MLP_MID
    params = I.init_params(wl, 44)
    x, y = I.make_batch(wl, 44, 1)
    q0 = _q0(wl.vocab, 34)
    hw = _head_index(wl)
    # a non-finite logit in the second shard's columns: that shard latches
    # BOM_ENONFINITE in its first part, the others BOM_ESHARD in their middle
    # part through its NaN row parts; q stays as it was everywhere
    pb = list(params)
    pb[hw] = params[hw].copy()
    pb[hw][700] = I.bf16_bits(np.full(wl.d_model, np.inf, dtype=np.float32))
    shards = _run_vshards(wl, pb, x, y, q0, 2, [500], check=False)
    assert shards[0]["stats"]["code"] == B.BOM_ESHARD
    assert shards[1]["stats"]["code"] == B.BOM_ENONFINITE
    for s in shards:
        assert np.array_equal(s["q"], q0[s["a"]:s["b"]].astype(np.float64))
        assert s["stats_end"]["code"] == s["stats"]["code"]
    # a label beyond the whole vocabulary: every shard latches BOM_ELABEL
    yb = y.copy()
    yb[123] = wl.vocab
    shards = _run_vshards(wl, params, x, yb, q0, 2, [500], check=False)
    for s in shards:
        assert s["stats"]["code"] == B.BOM_ELABEL
        assert np.array_equal(s["q"], q0[s["a"]:s["b"]].astype(np.float64))
    # no supervised row at all: every shard latches BOM_EEMPTY
    ye = np.full_like(y, I.IGNORE_INDEX)
    shards = _run_vshards(wl, params, x, ye, q0, 2, [500], check=False)
    for s in shards:
        assert s["stats"]["code"] == B.BOM_EEMPTY


def test_host_checks_of_the_vocab_sharded_calls():
    wl = I.LM_MLP_SMALL
    g = G.GpuBom(wl, I.init_params(wl, 0))
    x, y = I.make_batch(wl, 0, 1)
    n = wl.n_rows
    xd, yd = G.to_dev(x), torch.from_numpy(y).to(G.DEV)
    part = torch.zeros(n + 1, dtype=torch.float32, device=G.DEV)
    parts = torch.zeros((2, n), dtype=torch.float32, device=G.DEV)
    dh = torch.zeros((n, wl.d_model), dtype=torch.float32, device=G.DEV)
    grads = [torch.empty_like(p) for p in g.params]
    V = wl.vocab

    def code(fn, *a):
        with pytest.raises(B.BomError) as e:
            fn(*a)
        return e.value.code

    h = g.model.h
    # a middle or last part without the earlier ones
    assert code(B.bom_step_vshard_mid, h, xd, yd, n, g.params, g.q, 1, parts, 2, grads, dh) == B.BOM_EINVAL
    assert code(B.bom_step_vshard_end, h, xd, yd, n, g.params, dh, grads) == B.BOM_EINVAL
    # this shard's columns must lie inside the vocabulary
    assert code(B.bom_step_vshard_begin, h, xd, yd, n, g.params, V - 1, 0, part) == B.BOM_EINVAL
    assert code(B.bom_step_vshard_begin, h, xd, yd, n, g.params, 2 * V, V + 1, part) == B.BOM_EINVAL
    assert code(B.bom_step_vshard_begin, h, xd, yd, n, g.params, 2 * V, -1, part) == B.BOM_EINVAL
    # a misaligned row part
    assert code(B.bom_step_vshard_begin, h, xd, yd, n, g.params, 2 * V, V, part.data_ptr() + 2) == B.BOM_ENOTSUP
    B.bom_step_vshard_begin(h, xd, yd, n, g.params, 2 * V, V, part)
    # a middle part of another size, no shards, no cotangent buffer with a backbone
    assert code(B.bom_step_vshard_mid, h, xd, yd, n - 1, g.params, g.q, 1, parts, 2, grads, dh) == B.BOM_EINVAL
    assert code(B.bom_step_vshard_mid, h, xd, yd, n, g.params, g.q, 1, parts, 0, grads, dh) == B.BOM_EINVAL
    assert code(B.bom_step_vshard_mid, h, xd, yd, n, g.params, g.q, 1, parts, 2, grads, None) == B.BOM_EINVAL
    torch.cuda.synchronize()
    # the diagnostic g / h mode has two cotangents: not with vocabulary shards
    gh = G.GpuBom(wl, I.init_params(wl, 0), out_mode=B.BOM_OUT_G_AND_H)
    assert code(B.bom_step_vshard_begin, gh.model.h, xd, yd, n, gh.params, 2 * V, 0, part) == B.BOM_EINVAL
    torch.cuda.synchronize()


@pytest.mark.parametrize("name", ["lm_head_wide", "lm_mlp_k1100"])
def test_one_shard_holding_the_whole_head_equals_bom_step_bit_for_bit(name):
    """With one shard the combine of the row parts is exact (M + log 1) and
    the fp32 cotangent part is rounded to the compute dtype once, as the whole
    step's epilogue rounds it, so the three parts run the whole step's
    arithmetic in the same order.  (Both workloads take the general task-space
    path: n V is above the small pass's limit.)"""
    wl = I.WORKLOADS[name]
    params = I.init_params(wl, 45)
    x, y = I.make_batch(wl, 45, 1)
    q0, t = _q0(wl.vocab, 35), 2
    head_only = len(wl.layers) == 0
    shards = _run_vshards(wl, params, x, y, q0, t, [], input_grad=head_only)
    g = G.GpuBom(wl, params)
    g.q.copy_(torch.from_numpy(q0))
    dx = None
    if head_only:
        dx = torch.empty((wl.n_rows, wl.d_in), dtype=torch.bfloat16, device=G.DEV)
        B.bom_set_input_grad(g.model.h, dx)
    out = g.step(x, y, t)
    s = shards[0]
    assert s["stats"]["n_t"] == out["stats"]["n_t"]
    assert s["stats"]["loss"] == out["stats"]["loss"]
    assert np.array_equal(s["q"], out["q"])
    for k in ("qhat", "s", "lse"):
        assert np.array_equal(s[k], out[k]), k
    for k, (a, b) in enumerate(zip(s["grads"], out["grads"])):
        assert torch.equal(a, b), k
    if head_only:
        assert torch.equal(s["dx"], dx)
