"""Data-parallel partition of the BOM step on CPU ranks (world size 2, gloo).

Rows (tokens) split across ranks.  Each rank forms the residuals of its shard,
then one all-reduce of the column sums of R and of the integer N_t partial
gives every rank the same s_t, after which q_t updates redundantly.  With the
global qhat and N_t, each rank back-propagates its own rows; a second
all-reduce of the per-tensor partial gradients equals the full-batch u.  The
oracle's full-batch step is the reference (bit-exact counts, fp64 sums)."""
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
