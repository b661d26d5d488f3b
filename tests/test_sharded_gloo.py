"""Partitions of the BOM step on CPU ranks (world size 2, gloo).

Data parallel: rows (tokens) split across ranks.  Each rank forms the
residuals of its shard, then one all-reduce of the column sums of R and of the
integer N_t partial gives every rank the same s_t, after which q_t updates
redundantly.  With the global qhat and N_t, each rank back-propagates its own
rows; a second all-reduce of the per-tensor partial gradients equals the
full-batch u.

Vocabulary parallel (the head's output columns split across ranks): each rank
computes its logit columns, the per-row (max, sum exp) pairs are combined
across ranks into the row log-sum-exp, and s_t, q_t and qhat_t then live
sharded with no exchange.  The head weight gradient is local to the shard;
the head-input cotangent is the all-reduced sum of the shards' R W and
broadcast-row terms.

The oracle's full-batch step is the reference (bit-exact counts, fp64 sums)."""
import os
import socket

import numpy as np
import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

import oracle as O
from paper_2609_36738_gb300 import inputs as I
from tests import _indep as X

WL = I.LM_MLP_SMALL
LAM, B1, T = 0.5, 0.9, 2


def _free_port():
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    p = s.getsockname()[1]
    s.close()
    return p


def _rank_main(rank, world, port, out_dir):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        layers = X.oracle_layers(WL)
        params = X.params_f64(WL, I.init_params(WL, 4))
        xb, y = I.make_batch(WL, 4, 1)
        x = X.x_f64(WL, xb)
        rows = np.array_split(np.arange(WL.n_rows), world)[rank]
        q_prev = np.random.default_rng(5).standard_normal(WL.vocab) * 0.01
        q_prev -= q_prev.mean()
        # shard-local forward and residual column sums
        Z, saved = O.forward(layers, WL.head_bias, params, x[rows])
        valid = y[rows] != I.IGNORE_INDEX
        R = O.residuals(Z, y[rows], valid)
        colsum = torch.tensor(R.sum(axis=0))
        n_t = torch.tensor([int(valid.sum())], dtype=torch.int64)
        dist.all_reduce(colsum)
        dist.all_reduce(n_t)
        n_t = int(n_t.item())
        s = colsum.numpy() / n_t
        q, qhat = O.ema_update(q_prev, s, T, B1)
        # shard-local backward of the global-normalised mixed cotangent
        dZ = ((1 - LAM) * R + LAM * valid[:, None] * qhat[None, :]) / n_t
        grads, _, _ = O.backward(layers, WL.head_bias, params, saved, dZ)
        flat = torch.tensor(np.concatenate([g.ravel() for g in grads]))
        dist.all_reduce(flat)
        np.save(os.path.join(out_dir, f"rank{rank}.npy"),
                np.concatenate([[n_t], s, q, flat.numpy()]))
    finally:
        dist.destroy_process_group()


def test_two_rank_data_parallel_step_equals_full_batch(tmp_path):
    world = 2
    mp.spawn(_rank_main, args=(world, _free_port(), str(tmp_path)), nprocs=world, join=True)
    layers = X.oracle_layers(WL)
    params = X.params_f64(WL, I.init_params(WL, 4))
    xb, y = I.make_batch(WL, 4, 1)
    q_prev = np.random.default_rng(5).standard_normal(WL.vocab) * 0.01
    q_prev -= q_prev.mean()
    ref = O.bom_step(layers, WL.head_bias, params, X.x_f64(WL, xb), y, q_prev, T, lam=LAM, beta1=B1)
    u_ref = np.concatenate([u.ravel() for u in ref["u"]])
    V = WL.vocab
    outs = [np.load(tmp_path / f"rank{r}.npy") for r in range(world)]
    for o in outs:
        assert int(o[0]) == ref["n_t"]                      # integer count: exact
        assert X.rel_l2(o[1:1 + V], ref["s"]) < 1e-14
        assert X.rel_l2(o[1 + V:1 + 2 * V], ref["q"]) < 1e-14
        assert X.rel_l2(o[1 + 2 * V:], u_ref) < 1e-12
    # every rank holds the same state after the exchange
    assert np.array_equal(outs[0], outs[1])


WL_HEAD = I.LM_HEAD_SMALL


def _vocab_rank_main(rank, world, port, out_dir):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        wl = WL_HEAD
        W = X.params_f64(wl, I.init_params(wl, 6))[0]
        xb, y = I.make_batch(wl, 6, 1)
        H = X.x_f64(wl, xb)
        cols = np.array_split(np.arange(wl.vocab), world)[rank]
        q_prev = np.random.default_rng(8).standard_normal(wl.vocab) * 0.01
        Zl = H @ W[cols].T                                   # this rank's logit columns
        valid = y != I.IGNORE_INDEX
        n_t = int(valid.sum())                               # labels are replicated: no exchange
        # row log-sum-exp from the shards' (max, sum exp) pairs
        m_loc = torch.tensor(Zl.max(axis=1))
        m_all = m_loc.clone()
        dist.all_reduce(m_all, op=dist.ReduceOp.MAX)
        se = torch.tensor(np.exp(Zl - m_all.numpy()[:, None]).sum(axis=1))
        dist.all_reduce(se)
        lse = m_all.numpy() + np.log(se.numpy())
        P = np.exp(Zl - lse[:, None])
        own = (y[:, None] == cols[None, :]) & valid[:, None]
        R = np.where(valid[:, None], P - own, 0.0)
        s = R.sum(axis=0) / n_t                              # sharded s_t: no exchange
        q, qhat = O.ema_update(q_prev[cols], s, T, B1)
        dZ = ((1 - LAM) * R + LAM * valid[:, None] * qhat[None, :]) / n_t
        gW = dZ.T @ H                                         # local rows of the head gradient
        dH = torch.tensor(dZ @ W[cols])
        dist.all_reduce(dH)                                   # head-input cotangent
        np.save(os.path.join(out_dir, f"vrank{rank}.npy"),
                np.concatenate([[n_t], cols, s, q, gW.ravel(), dH.numpy().ravel()]))
    finally:
        dist.destroy_process_group()


def test_two_rank_vocabulary_parallel_head_equals_full_batch(tmp_path):
    world = 2
    mp.spawn(_vocab_rank_main, args=(world, _free_port(), str(tmp_path)), nprocs=world, join=True)
    wl = WL_HEAD
    params = X.params_f64(wl, I.init_params(wl, 6))
    xb, y = I.make_batch(wl, 6, 1)
    q_prev = np.random.default_rng(8).standard_normal(wl.vocab) * 0.01
    ref = O.bom_step(X.oracle_layers(wl), wl.head_bias, params, X.x_f64(wl, xb), y, q_prev, T, lam=LAM, beta1=B1)
    d = wl.d_in
    dHs = []
    for r in range(world):
        o = np.load(tmp_path / f"vrank{r}.npy")
        assert int(o[0]) == ref["n_t"]
        cols = np.array_split(np.arange(wl.vocab), world)[r]
        k = 1 + cols.size
        assert np.array_equal(o[1:k].astype(np.int64), cols)
        s, q = o[k:k + cols.size], o[k + cols.size:k + 2 * cols.size]
        assert X.rel_l2(s, ref["s"][cols]) < 1e-13
        assert X.rel_l2(q, ref["q"][cols]) < 1e-13
        g0 = k + 2 * cols.size
        gW = o[g0:g0 + cols.size * d].reshape(cols.size, d)
        assert X.rel_l2(gW, ref["u"][0][cols]) < 1e-12
        dHs.append(o[g0 + cols.size * d:])
    assert X.rel_l2(dHs[0], ref["dX_u"].ravel()) < 1e-12
    assert np.array_equal(dHs[0], dHs[1])


class _OracleShardCalls:
    """Stands in for the library's two row-shard calls on CPU ranks: the same
    exchange-vector layout (column sums of R, CE sum, N_t, error flag) and the
    same gradient shares, computed by the oracle, so that bench.dp_step's
    order of calls and collectives runs on gloo ranks without a GPU."""

    def __init__(self, wl, params64, lam, beta1):
        self.wl, self.p, self.lam, self.beta1 = wl, params64, lam, beta1
        self.layers = X.oracle_layers(wl)
        self.calls = []

    def bom_step_shard_begin(self, h, x, y, n, params, xch, stream=None):
        self.calls.append("begin")
        V = self.wl.vocab
        Z, saved = O.forward(self.layers, self.wl.head_bias, self.p, x)
        valid = y != I.IGNORE_INDEX
        R = O.residuals(Z, y, valid)
        lse = O.log_sum_exp_rows(Z)
        ce = float(np.sum((lse - Z[np.arange(len(y)), np.where(valid, y, 0)])[valid]))
        xch[:V] = torch.from_numpy(R.sum(axis=0))
        xch[V] = ce
        xch[V + 1] = float(valid.sum())
        xch[V + 2] = 0.0
        self.state = (saved, R, valid)

    def bom_step_shard_end(self, h, x, y, n, params, q, t, xch, grads, h_out, stream=None):
        self.calls.append("end")
        V = self.wl.vocab
        saved, R, valid = self.state
        n_t = float(xch[V + 1])
        s = xch[:V].numpy() / n_t
        q_new, qhat = O.ema_update(q.numpy().copy(), s, t, self.beta1)
        q.copy_(torch.from_numpy(q_new))
        dZ = ((1 - self.lam) * R + self.lam * valid[:, None] * qhat[None, :]) / n_t
        gr, _, _ = O.backward(self.layers, self.wl.head_bias, self.p, saved, dZ)
        for g, v in zip(grads, gr):
            g.copy_(torch.from_numpy(np.asarray(v).reshape(g.shape)))


def _bench_dp_rank_main(rank, world, port, out_dir):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        import bench
        params = X.params_f64(WL, I.init_params(WL, 4))
        xb, y = I.make_batch(WL, 4, 1)
        x = X.x_f64(WL, xb)
        rows = np.array_split(np.arange(WL.n_rows), world)[rank]
        q_prev = np.random.default_rng(5).standard_normal(WL.vocab) * 0.01
        q_prev -= q_prev.mean()
        lib = _OracleShardCalls(WL, params, LAM, B1)
        sizes = [p.size for p in params]
        flat = torch.zeros(sum(sizes), dtype=torch.float64)
        views = [v.view(p.shape) for v, p in zip(torch.split(flat, sizes), params)]
        xch = torch.full((WL.vocab + 3,), float("nan"), dtype=torch.float64)
        q = torch.from_numpy(q_prev.copy())
        order = []

        def allreduce(tensor):
            order.append("allreduce")
            dist.all_reduce(tensor)

        bench.dp_step(lib, None, x[rows], y[rows], rows.size, params, q, T, xch, views, flat, allreduce)
        calls = [c for c in lib.calls]
        np.save(os.path.join(out_dir, f"dp{rank}.npy"), np.concatenate([[xch[WL.vocab + 1].item()], q.numpy(),
                                                                         flat.numpy()]))
        with open(os.path.join(out_dir, f"dp{rank}.txt"), "w") as f:
            f.write(" ".join(calls) + " | " + " ".join(order))
    finally:
        dist.destroy_process_group()


def test_bench_data_parallel_step_on_two_gloo_ranks(tmp_path):
    """bench.dp_step, the data-parallel step of bench.py --gpus N: begin, the
    sum of the exchange vectors, end, the sum of the gradient shares.  On two
    gloo ranks with the oracle standing in for the library's shard calls,
    every rank ends with the whole batch's N_t, q and u."""
    world = 2
    mp.spawn(_bench_dp_rank_main, args=(world, _free_port(), str(tmp_path)), nprocs=world, join=True)
    layers = X.oracle_layers(WL)
    params = X.params_f64(WL, I.init_params(WL, 4))
    xb, y = I.make_batch(WL, 4, 1)
    q_prev = np.random.default_rng(5).standard_normal(WL.vocab) * 0.01
    q_prev -= q_prev.mean()
    ref = O.bom_step(layers, WL.head_bias, params, X.x_f64(WL, xb), y, q_prev, T, lam=LAM, beta1=B1)
    u_ref = np.concatenate([u.ravel() for u in ref["u"]])
    V = WL.vocab
    outs = [np.load(tmp_path / f"dp{r}.npy") for r in range(world)]
    for r, o in enumerate(outs):
        assert int(o[0]) == ref["n_t"]
        assert X.rel_l2(o[1:1 + V], ref["q"]) < 1e-14
        assert X.rel_l2(o[1 + V:], u_ref) < 1e-12
        assert (tmp_path / f"dp{r}.txt").read_text() == "begin end | allreduce allreduce"
    assert np.array_equal(outs[0], outs[1])


def _vocab_lse_parts_rank_main(rank, world, port, out_dir):
    """The exchange bom_step_vshard_begin / _mid use: each rank's part of a
    row's log-sum-exp over its own columns, all-gathered in rank order, then
    combined on every rank as M + log sum_r exp(part_r - M)."""
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        wl = WL_HEAD
        W = X.params_f64(wl, I.init_params(wl, 7))[0]
        xb, y = I.make_batch(wl, 7, 1)
        H = X.x_f64(wl, xb)
        cols = np.array_split(np.arange(wl.vocab), world)[rank]
        Zl = H @ W[cols].T
        part = torch.tensor(O.log_sum_exp_rows(Zl))          # this rank's part of every row
        parts = [torch.zeros_like(part) for _ in range(world)]
        dist.all_gather(parts, part)
        P = torch.stack(parts).numpy()                         # [world, n], rank order
        M = P.max(axis=0)
        lse = M + np.log(np.exp(P - M[None, :]).sum(axis=0))
        valid = y != I.IGNORE_INDEX
        own = valid & (y >= cols[0]) & (y <= cols[-1])
        ce_part = float(np.sum((lse - Zl[np.arange(len(y)), np.where(own, y - cols[0], 0)])[own]))
        np.save(os.path.join(out_dir, f"lrank{rank}.npy"), np.concatenate([lse, [ce_part]]))
    finally:
        dist.destroy_process_group()


def test_vocabulary_lse_parts_combine_to_the_whole_row_and_the_ce_parts_to_the_loss(tmp_path):
    world = 3
    mp.spawn(_vocab_lse_parts_rank_main, args=(world, _free_port(), str(tmp_path)), nprocs=world, join=True)
    wl = WL_HEAD
    params = X.params_f64(wl, I.init_params(wl, 7))
    xb, y = I.make_batch(wl, 7, 1)
    Z, _ = O.forward(X.oracle_layers(wl), wl.head_bias, params, X.x_f64(wl, xb))
    valid, n_t = O.supervised_set(y, wl.vocab)
    ce, lse = O.cross_entropy(Z, y, valid, n_t)
    outs = [np.load(tmp_path / f"lrank{r}.npy") for r in range(world)]
    for o in outs:
        assert X.rel_l2(o[:-1], lse) < 1e-14
        assert np.array_equal(o[:-1], outs[0][:-1])            # every rank combines the same floats
    # each supervised row's CE lies in exactly one rank's part; the parts add up to the loss
    assert abs(sum(o[-1] for o in outs) / n_t - ce) < 1e-12 * abs(ce)


class _OracleVocabCalls:
    """Stands in for the library's three vocabulary-shard calls on CPU ranks,
    computed by the oracle: this rank's log-sum-exp part, then (from every
    rank's parts) its residuals, s_t, q_t, head rows of u and its part of the
    head's input cotangent, then the backbone's backward from the summed
    cotangent (the oracle's reverse pass with an identity head, so that the
    cotangent of the head input is the given sum)."""

    def __init__(self, wl, params64, cols, lam, beta1):
        self.wl, self.p, self.cols, self.lam, self.beta1 = wl, params64, cols, lam, beta1
        self.layers = X.oracle_layers(wl)
        self.hw = len(params64) - (2 if wl.head_bias else 1)
        self.calls = []

    def bom_step_vshard_begin(self, h, x, y, n, params, v_total, v_first, lse_part, stream=None):
        self.calls.append("begin")
        assert v_first == self.cols[0] and v_total == self.wl.vocab
        Z, saved = O.forward(self.layers, self.wl.head_bias, self.p, x)
        self.Zr, self.saved = Z[:, self.cols], saved
        lse_part.copy_(torch.from_numpy(O.log_sum_exp_rows(self.Zr)))

    def bom_step_vshard_mid(self, h, x, y, n, params, q, t, lse_parts, n_shards, grads, dh, stream=None):
        self.calls.append("mid")
        P = lse_parts.numpy()
        assert P.shape[0] == n_shards
        M = P.max(axis=0)
        lse = M + np.log(np.exp(P - M[None, :]).sum(axis=0))
        valid = y != I.IGNORE_INDEX
        n_t = int(valid.sum())
        onehot = (y[:, None] == self.cols[None, :]) & valid[:, None]
        R = np.where(valid[:, None], np.exp(self.Zr - lse[:, None]) - onehot, 0.0)
        s = R.sum(axis=0) / n_t
        q_new, qhat = O.ema_update(q.numpy().copy(), s, t, self.beta1)
        q.copy_(torch.from_numpy(q_new))
        dZ = ((1 - self.lam) * R + self.lam * valid[:, None] * qhat[None, :]) / n_t
        grads[self.hw].copy_(torch.from_numpy(dZ.T @ self.saved[1]))
        dh.copy_(torch.from_numpy(dZ @ self.p[self.hw][self.cols]))

    def bom_step_vshard_end(self, h, x, y, n, params, dh_sum, grads, stream=None):
        self.calls.append("end")
        d = self.saved[1].shape[1]
        gr, _, _ = O.backward(self.layers, False, list(self.p[:self.hw]) + [np.eye(d)], self.saved, dh_sum.numpy())
        for k in range(self.hw):
            grads[k].copy_(torch.from_numpy(gr[k]))


def _bench_vocab_rank_main(rank, world, port, out_dir):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        import bench
        wl = WL
        params = X.params_f64(wl, I.init_params(wl, 8))
        xb, y = I.make_batch(wl, 8, 1)          # every rank holds the whole batch
        x = X.x_f64(wl, xb)
        cols = np.array_split(np.arange(wl.vocab), world)[rank]
        q_prev = np.random.default_rng(9).standard_normal(wl.vocab) * 0.01
        lib = _OracleVocabCalls(wl, params, cols, LAM, B1)
        n, d = wl.n_rows, wl.d_model
        grads = [torch.zeros(p.shape, dtype=torch.float64) for p in params]
        grads[lib.hw] = torch.zeros((cols.size, d), dtype=torch.float64)
        q = torch.from_numpy(q_prev[cols].copy())
        lse_part = torch.zeros(n, dtype=torch.float64)
        lse_parts = torch.zeros((world, n), dtype=torch.float64)
        dh = torch.zeros((n, d), dtype=torch.float64)
        order = []

        def allgather(out, part):
            order.append("allgather")
            dist.all_gather(list(out.unbind(0)), part)

        def allreduce(tensor):
            order.append("allreduce")
            dist.all_reduce(tensor)

        bench.vocab_step(lib, None, x, y, n, params, wl.vocab, int(cols[0]), q, T, lse_part, lse_parts, dh, grads,
                         allgather, allreduce)
        np.save(os.path.join(out_dir, f"vb{rank}.npy"),
                np.concatenate([q.numpy()] + [g.numpy().ravel() for g in grads]))
        with open(os.path.join(out_dir, f"vb{rank}.txt"), "w") as f:
            f.write(" ".join(lib.calls) + " | " + " ".join(order))
    finally:
        dist.destroy_process_group()


def test_bench_vocabulary_parallel_step_on_two_gloo_ranks(tmp_path):
    """bench.vocab_step, the vocabulary-parallel step of bench.py --parallel
    vocab: begin, the all-gather of the row log-sum-exp parts, mid, the
    all-reduce of the head's input cotangent, end.  On two gloo ranks with the
    oracle standing in for the library's three calls, every rank ends with its
    entries of q and rows of the head's u, and the whole batch's u of every
    backbone tensor."""
    world = 2
    mp.spawn(_bench_vocab_rank_main, args=(world, _free_port(), str(tmp_path)), nprocs=world, join=True)
    wl = WL
    layers = X.oracle_layers(wl)
    params = X.params_f64(wl, I.init_params(wl, 8))
    xb, y = I.make_batch(wl, 8, 1)
    q_prev = np.random.default_rng(9).standard_normal(wl.vocab) * 0.01
    ref = O.bom_step(layers, wl.head_bias, params, X.x_f64(wl, xb), y, q_prev, T, lam=LAM, beta1=B1)
    hw = len(params) - (2 if wl.head_bias else 1)
    backbone = np.concatenate([ref["u"][k].ravel() for k in range(hw)])
    outs = []
    for r in range(world):
        cols = np.array_split(np.arange(wl.vocab), world)[r]
        o = np.load(tmp_path / f"vb{r}.npy")
        assert X.rel_l2(o[:cols.size], ref["q"][cols]) < 1e-13
        nb = backbone.size
        assert X.rel_l2(o[cols.size:cols.size + nb], backbone) < 1e-12
        assert X.rel_l2(o[cols.size + nb:], ref["u"][hw][cols].ravel()) < 1e-12
        assert (tmp_path / f"vb{r}.txt").read_text() == "begin mid end | allgather allreduce"
        outs.append(o[cols.size:cols.size + nb])
    assert np.array_equal(outs[0], outs[1])   # the backbone's u is the same on every rank
