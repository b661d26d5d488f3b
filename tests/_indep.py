"""Independent fp64 re-implementations used to pin the oracle.

These do not call the oracle: the forward pass is written with torch.nn.functional
(a separate code path from the oracle's numpy), gradients come from torch
autograd, and Jacobians from central finite differences of that forward.
"""
from __future__ import annotations

import numpy as np
import torch
import torch.nn.functional as F

from paper_2609_36738_gb300 import inputs as I



def oracle_layers(wl: I.Workload):
    return [(l.kind, l.d_in, l.d_out, l.has_bias) for l in wl.layers]


def params_f64(wl: I.Workload, params):
    if wl.dtype == "bf16":
        return [I.bf16_to_f64(p) for p in params]
    return [np.asarray(p, dtype=np.float64) for p in params]


def x_f64(wl: I.Workload, x):
    return I.bf16_to_f64(x) if wl.dtype == "bf16" else np.asarray(x, dtype=np.float64)


def torch_forward(wl: I.Workload, params, X):
    """Logits through torch.nn.functional ops (fp64)."""
    it = iter(params)
    x = X
    for l in wl.layers:
        if l.kind == I.SWIGLU:
            wg, wu, wd = next(it), next(it), next(it)
            x = x + F.linear(F.silu(F.linear(x, wg)) * F.linear(x, wu), wd)
        elif l.kind == I.RMSNORM:
            x = F.rms_norm(x, (l.d_in,), weight=next(it), eps=1e-6)
        else:
            w = next(it)
            b = next(it) if l.has_bias else None
            x = F.linear(x, w, b)
            if l.kind == I.LINEAR_GELU:
                x = F.gelu(x, approximate="none")
    hw = next(it)
    hb = next(it) if wl.head_bias else None
    return F.linear(x, hw, hb)


def autograd_mix(wl, params_np, X_np, labels, qhat, lam, ignore_index=-100):
    """Gradient of L_mix = (1-lam) CE + lam/N_t sum_i <z_i, qhat> via autograd."""
    ps = [torch.tensor(p, requires_grad=True) for p in params_np]
    X = torch.tensor(X_np, requires_grad=True)
    Z = torch_forward(wl, ps, X)
    y = torch.tensor(np.asarray(labels, dtype=np.int64))
    valid = y != ignore_index
    n_t = int(valid.sum())
    ce = F.cross_entropy(Z, y, ignore_index=ignore_index, reduction="sum") / n_t
    sur = (Z[valid] @ torch.tensor(qhat)).sum() / n_t
    loss = (1 - lam) * ce + lam * sur
    grads = torch.autograd.grad(loss, ps + [X])
    autograd_mix.last_dX = grads[-1].numpy()
    return [g.numpy() for g in grads[:-1]], float(ce.detach())


def fd_jacobians(wl, params_np, X_np, eps=1e-6):
    """Per-example Jacobians J[i] = d z_i / d theta (d_out x P), central differences."""
    flat = np.concatenate([p.ravel() for p in params_np])
    shapes = [p.shape for p in params_np]
    X = torch.tensor(X_np)

    def unflat(v):
        out, o = [], 0
        for s in shapes:
            n = int(np.prod(s))
            out.append(torch.tensor(v[o:o + n].reshape(s)))
            o += n
        return out

    n, c = X_np.shape[0], wl.vocab
    J = np.zeros((n, c, flat.size))
    v = flat.copy()
    with torch.no_grad():
        for k in range(flat.size):
            v[k] = flat[k] + eps
            zp = torch_forward(wl, unflat(v), X).numpy()
            v[k] = flat[k] - eps
            zm = torch_forward(wl, unflat(v), X).numpy()
            v[k] = flat[k]
            J[:, :, k] = (zp - zm) / (2 * eps)
    return J


def unflatten(vec, params_np):
    out, o = [], 0
    for p in params_np:
        out.append(vec[o:o + p.size].reshape(p.shape))
        o += p.size
    return out


def rel_l2(a, b):
    a = np.asarray(a, dtype=np.float64).ravel()
    b = np.asarray(b, dtype=np.float64).ravel()
    nb = np.linalg.norm(b)
    return float(np.linalg.norm(a - b) / (nb if nb > 0 else 1.0))
