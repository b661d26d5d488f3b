"""Plain fp64 CPU oracle of one BOM step and of the BOM-AdamW update.

TEST INFRASTRUCTURE ONLY.  Nothing on the product path may import, call or
execute this module: only ``tests/``, ``__graft_entry__.smoke()`` and the
CPU-baseline / reference legs of ``bench.py`` use it.  It shares no code with
the CUDA path (no kernels, headers, helpers, tables or constants); the two
meet only in the seeded input generator, which holds none of the method's
arithmetic.

Everything is numpy float64.  Inputs arrive as the exact values the GPU sees
(fp32 values, or bf16 values already expanded), promoted to float64, so only
the compute precision differs between the two sides.

What it computes (paper: "Backpropagated Output Momentum", Algorithm 1 in the
per-dataset-results appendix, with the equations of Section 3):

  1. supervised set I_t = rows whose label is not ``ignore_index``,
     N_t = |I_t| > 0 (Algorithm 1, first step; LM construction appendix);
  2. r_i = softmax(z_i) - onehot(y_i),  s_t = N_t^-1 sum_{i in I_t} r_i
     (Algorithm 1; Section 3.2, "Formal update");
  3. q_t = beta1 q_{t-1} + (1 - beta1) s_t,  qhat_t = q_t / (1 - beta1^t)
     (Section 3.2, the EMA equation);
  4. L_mix = (1 - lambda) L_CE + lambda N_t^-1 sum_i <z_i, qhat_t>
     (Eq. mix-objective); its gradient u = (1 - lambda) g + lambda Jbar^T qhat
     (Eq. mix-gradient).  The oracle back-propagates the logit cotangent of
     L_mix by hand:  dL_mix/dz_i = N_t^-1 [(1 - lambda) r_i + lambda qhat_t]
     for i in I_t and 0 otherwise.  g (cotangent r_i / N_t) and
     h = Jbar^T qhat (cotangent qhat / N_t) are also returned separately;
  5. v = beta2 v + (1 - beta2) u^2,  vhat = v / (1 - beta2^t)
     (Section 3.4, the second-moment equation);
  6. theta <- (1 - eta omega) theta - eta u / (sqrt(vhat) + eps)
     (Section 3.4 update equation; Algorithm 1, last step).  No first-moment
     bias correction is applied to u (Section 3.5, "The substitution");
  7. drift telemetry and the own-step control (Section 3.3, Eq.
     drift-telemetry; stale-control and drift-measurement appendices): the
     own-step projection Jbar_t^T s_t, its EMA M_t with Mhat_t, the cosine and
     relative size of Mhat_t - h_t, and the within-batch cancellation ratio;
  8. BOM-Adam-mini (Section 3.5, composition with Adam-mini): the update with
     one second-moment scalar shared by each block of a tensor;
  9. global-norm clipping of u before the update (pretraining-parameters and
     convergence appendices).

Backbone layers supported (shapes of the paper's settings; see the workload
module): Linear, Linear+GELU (exact erf form), the SwiGLU MLP sublayer
x <- x + W_d (SiLU(W_g x) * W_u x) and RMSNorm x / sqrt(mean x^2 + 1e-6) * gamma
(the norm tensors of the language-model setting).  The head is Linear
d -> d_out, with an optional bias.

Every function here is pinned by ``tests/test_oracle_pins.py`` against facts
the paper or mathematics fix (finite-difference Jacobians and the exact batch
decomposition, an independent autograd implementation, the EMA closed form of
Lemma 2, the beta1 = 0 and lambda = 0 reductions, AdamW with beta1 = 0, the
output-bias closed form and the zero-sum invariant); the telemetry functions
by ``tests/test_oracle_telemetry_pins.py`` (finite-difference Jbar^T s, no drift
at t = 1 and for a linear model on a fixed batch, Mhat = qhat on the head bias,
closed forms and a brute-force loop for the statistics).
"""
from __future__ import annotations

import math
from typing import Dict, List, Sequence, Tuple

import numpy as np
from scipy.special import erf as _erf

F64 = np.float64


class OracleError(Exception):
    pass


class LabelError(OracleError):
    """A label outside [0, d_out) that is not the ignore index."""


class EmptyError(OracleError):
    """N_t = 0: Algorithm 1 requires at least one supervised output."""


# --------------------------------------------------------------------------
# Activations (exact GELU; SiLU = x * sigmoid(x))
# --------------------------------------------------------------------------
def gelu(x):
    return 0.5 * x * (1.0 + _erf(x / math.sqrt(2.0)))


def gelu_prime(x):
    # d/dx [x Phi(x)] = Phi(x) + x phi(x)
    Phi = 0.5 * (1.0 + _erf(x / math.sqrt(2.0)))
    phi = np.exp(-0.5 * x * x) / math.sqrt(2.0 * math.pi)
    return Phi + x * phi


def sigmoid(x):
    return 1.0 / (1.0 + np.exp(-x))


def silu(x):
    return x * sigmoid(x)


def silu_prime(x):
    sg = sigmoid(x)
    return sg * (1.0 + x * (1.0 - sg))


# RMSNorm (the norm tensors of the paper's Qwen3 language models, weight decay
# 0): y = x / sqrt(mean_j x_j^2 + eps) * gamma with the Qwen3 epsilon.
RMS_EPS = 1e-6


# --------------------------------------------------------------------------
# Model: layers are (kind, d_in, d_out, has_bias) with kind in
# {"linear", "linear_gelu", "swiglu", "rmsnorm"}; parameters are listed per
# layer (W [d_out, d_in], b [d_out]), (W_gate [ffn, d], W_up [ffn, d],
# W_down [d, ffn]) or (gamma [d]), followed by the head (W [d_out, d],
# optional b).
# --------------------------------------------------------------------------
def _split_params(layers, head_bias, params):
    it = iter(params)
    per_layer = []
    for kind, d_in, d_out, has_bias in layers:
        if kind == "swiglu":
            per_layer.append((next(it), next(it), next(it)))
        elif kind == "rmsnorm":
            per_layer.append((next(it),))
        else:
            w = next(it)
            b = next(it) if has_bias else None
            per_layer.append((w, b))
    hw = next(it)
    hb = next(it) if head_bias else None
    rest = list(it)
    if rest:
        raise OracleError("too many parameter tensors")
    return per_layer, (hw, hb)


def forward(layers, head_bias, params, X):
    """Logits Z = f(theta; X) and the saved activations of every layer."""
    per_layer, (hw, hb) = _split_params(layers, head_bias, params)
    x = np.asarray(X, dtype=F64)
    tape = []
    for (kind, d_in, d_out, has_bias), p in zip(layers, per_layer):
        if kind == "swiglu":
            wg, wu, wd = p
            G = x @ wg.T
            U = x @ wu.T
            A = silu(G) * U
            y = x + A @ wd.T
            tape.append(("swiglu", x, G, U, A))
            x = y
        elif kind == "rmsnorm":
            (gamma,) = p
            r = 1.0 / np.sqrt(np.mean(x * x, axis=1, keepdims=True) + RMS_EPS)
            xhat = x * r
            tape.append(("rmsnorm", x, r, xhat))
            x = xhat * gamma
        else:
            w, b = p
            pre = x @ w.T
            if b is not None:
                pre = pre + b
            tape.append((kind, x, pre))
            x = gelu(pre) if kind == "linear_gelu" else pre
    Z = x @ hw.T
    if hb is not None:
        Z = Z + hb
    return Z, (tape, x)


def backward(layers, head_bias, params, saved, dZ):
    """Vector-Jacobian product of the logit cotangent dZ through the network.

    Returns (grads per parameter tensor in interface order, cotangent of the
    head input, cotangent of the network input X)."""
    per_layer, (hw, hb) = _split_params(layers, head_bias, params)
    tape, h_last = saved
    dZ = np.asarray(dZ, dtype=F64)
    g_hw = dZ.T @ h_last
    g_hb = dZ.sum(axis=0) if hb is not None else None
    dx = dZ @ hw
    dx_head = dx
    grads_rev: List[np.ndarray] = []
    if hb is not None:
        grads_rev.append(g_hb)
    grads_rev.append(g_hw)
    for li in range(len(layers) - 1, -1, -1):
        kind = layers[li][0]
        rec = tape[li]
        if kind == "swiglu":
            wg, wu, wd = per_layer[li]
            _, x, G, U, A = rec
            dy = dx
            g_wd = dy.T @ A
            dA = dy @ wd
            dG = dA * U * silu_prime(G)
            dU = dA * silu(G)
            g_wg = dG.T @ x
            g_wu = dU.T @ x
            dx = dy + dG @ wg + dU @ wu
            grads_rev.extend([g_wd, g_wu, g_wg])
        elif kind == "rmsnorm":
            (gamma,) = per_layer[li]
            _, x, r, xhat = rec
            grads_rev.append((dx * xhat).sum(axis=0))
            dxhat = dx * gamma
            # d/dx of x r(x): r (dxhat - xhat mean_j(dxhat_j xhat_j))
            dx = r * (dxhat - xhat * np.mean(dxhat * xhat, axis=1, keepdims=True))
        else:
            w, b = per_layer[li]
            _, x, pre = rec
            dpre = dx * gelu_prime(pre) if kind == "linear_gelu" else dx
            g_w = dpre.T @ x
            if b is not None:
                grads_rev.append(dpre.sum(axis=0))
            grads_rev.append(g_w)
            dx = dpre @ w
    return grads_rev[::-1], dx_head, dx


# --------------------------------------------------------------------------
# Task-space quantities (Algorithm 1, residual / EMA / objective steps)
# --------------------------------------------------------------------------
def supervised_set(labels, d_out, ignore_index=-100):
    """Boolean mask of I_t and N_t; raises on bad labels or N_t = 0."""
    y = np.asarray(labels, dtype=np.int64)
    valid = y != ignore_index
    bad = valid & ((y < 0) | (y >= d_out))
    if bad.any():
        raise LabelError(f"{int(bad.sum())} labels outside [0, {d_out})")
    n_t = int(valid.sum())
    if n_t == 0:
        raise EmptyError("no supervised outputs in the batch (N_t = 0)")
    return valid, n_t


def log_sum_exp_rows(Z):
    m = Z.max(axis=1, keepdims=True)
    return (m + np.log(np.exp(Z - m).sum(axis=1, keepdims=True)))[:, 0]


def softmax_rows(Z):
    m = Z.max(axis=1, keepdims=True)
    e = np.exp(Z - m)
    return e / e.sum(axis=1, keepdims=True)


def residuals(Z, labels, valid):
    """r_i = softmax(z_i) - onehot(y_i) on supervised rows, 0 elsewhere."""
    R = softmax_rows(np.asarray(Z, dtype=F64))
    rows = np.nonzero(valid)[0]
    R[rows, np.asarray(labels)[rows]] -= 1.0
    R[~valid] = 0.0
    return R


def batch_mean_residual(R, n_t):
    """s_t = N_t^-1 sum_{i in I_t} r_i (ignored rows of R are zero)."""
    return R.sum(axis=0) / n_t


def ema_update(q_prev, s, t, beta1):
    """q_t = beta1 q_{t-1} + (1 - beta1) s_t and qhat_t = q_t / (1 - beta1^t)."""
    q = beta1 * np.asarray(q_prev, dtype=F64) + (1.0 - beta1) * np.asarray(s, dtype=F64)
    qhat = q / (1.0 - beta1 ** t)
    return q, qhat


def cross_entropy(Z, labels, valid, n_t):
    lse = log_sum_exp_rows(Z)
    rows = np.nonzero(valid)[0]
    zy = Z[rows, np.asarray(labels)[rows]]
    return float((lse[rows] - zy).sum() / n_t), lse


def bom_step(layers, head_bias, params, X, labels, q_prev, t, lam=0.5, beta1=0.9,
             ignore_index=-100) -> Dict[str, object]:
    """One BOM step up to the update numerator (Algorithm 1, first five steps).

    Returns a dict with the logits ``Z``, row log-sum-exp ``lse``, ``ce``,
    ``n_t``, ``valid``, ``s``, ``q``, ``qhat`` and per-tensor lists ``g``, ``h``,
    ``u``, plus the head-input cotangents ``dx_g``, ``dx_h``, ``dx_u`` and the
    input cotangents ``dX_g``, ``dX_h``, ``dX_u``."""
    if t < 1:
        raise OracleError("t is 1-based")
    params = [np.asarray(p, dtype=F64) for p in params]
    Z, saved = forward(layers, head_bias, params, X)
    d_out = Z.shape[1]
    valid, n_t = supervised_set(labels, d_out, ignore_index)
    R = residuals(Z, labels, valid)
    s = batch_mean_residual(R, n_t)
    q, qhat = ema_update(q_prev, s, t, beta1)
    ce, lse = cross_entropy(Z, labels, valid, n_t)
    # Logit cotangents of the three objectives.
    d_g = R / n_t                                   # CE part: g
    d_h = valid[:, None] * qhat[None, :] / n_t      # surrogate part: Jbar^T qhat
    d_u = (1.0 - lam) * d_g + lam * d_h             # L_mix (Eq. mix-objective)
    g, dx_g, dX_g = backward(layers, head_bias, params, saved, d_g)
    h, dx_h, dX_h = backward(layers, head_bias, params, saved, d_h)
    u, dx_u, dX_u = backward(layers, head_bias, params, saved, d_u)
    return dict(Z=Z, lse=lse, ce=ce, n_t=n_t, valid=valid, R=R, s=s, q=q, qhat=qhat,
                g=g, h=h, u=u, dx_g=dx_g, dx_h=dx_h, dx_u=dx_u, dX_g=dX_g, dX_h=dX_h, dX_u=dX_u)


# --------------------------------------------------------------------------
# BOM-AdamW update (Section 3.4; Algorithm 1, last two steps)
# --------------------------------------------------------------------------
def bom_update(theta, u, v, lr, wd, t, beta2=0.999, eps=1e-8):
    """Returns (theta_new, v_new) in float64."""
    if t < 1:
        raise OracleError("t is 1-based")
    theta = np.asarray(theta, dtype=F64)
    u = np.asarray(u, dtype=F64)
    v_new = beta2 * np.asarray(v, dtype=F64) + (1.0 - beta2) * u * u
    vhat = v_new / (1.0 - beta2 ** t)
    theta_new = (1.0 - lr * wd) * theta - lr * u / (np.sqrt(vhat) + eps)
    return theta_new, v_new


def mix_numerator(g, h, lam):
    """u = (1 - lambda) g + lambda h (Eq. mix-gradient)."""
    return (1.0 - lam) * np.asarray(g, dtype=F64) + lam * np.asarray(h, dtype=F64)


def bom_update_gh(theta, g, h, v, lr, wd, lam, t, beta2=0.999, eps=1e-8):
    """Update from the separate supervised gradient g and reprojection h."""
    return bom_update(theta, mix_numerator(g, h, lam), v, lr, wd, t, beta2, eps)


# --------------------------------------------------------------------------
# Sampled head gradients (full-size checks where the full reverse pass is too
# slow in fp64).  Same formulas as `backward` for the head, restricted to a
# subset of output rows: with the L_mix logit cotangent
#   dZ = N_t^-1 [(1 - lambda) R + lambda 1_{I_t} qhat^T],
# the head weight gradient is dZ^T H and the head-input cotangent is dZ W.
# --------------------------------------------------------------------------
def mix_cotangent_rows(R, valid, qhat, n_t, lam, rows):
    """Rows `rows` of dZ (Eq. mix-objective, differentiated in the logits)."""
    rows = np.asarray(rows)
    return ((1.0 - lam) * R[rows] + lam * valid[rows, None] * np.asarray(qhat)[None, :]) / n_t


def head_weight_grad_rows(R, H, valid, qhat, n_t, lam, vocab_rows):
    """Rows `vocab_rows` of the head weight gradient dZ^T H."""
    vocab_rows = np.asarray(vocab_rows)
    dZ_cols = ((1.0 - lam) * R[:, vocab_rows] + lam * valid[:, None] * np.asarray(qhat)[None, vocab_rows]) / n_t
    return dZ_cols.T @ np.asarray(H, dtype=F64)


def head_input_grad_rows(R, W, valid, qhat, n_t, lam, token_rows):
    """Rows `token_rows` of the head-input cotangent dZ W."""
    return mix_cotangent_rows(R, valid, qhat, n_t, lam, token_rows) @ np.asarray(W, dtype=F64)


def mix_grad_rows(layers, head_bias, params, saved, R, valid, qhat, n_t, lam, rows):
    """Sampled output rows of u = (1 - lambda) g + lambda Jbar^T qhat for EVERY
    parameter tensor (Eq. mix-gradient), for full-size checks of a whole
    network where `backward` would form every weight gradient in full.

    The reverse pass is the one of `backward`, with the L_mix logit cotangent
    dZ = N_t^-1 [(1 - lambda) R + lambda 1_{I_t} qhat^T] (Eq. mix-objective,
    differentiated in the logits), walked from the head down:
      head input:  dZ W = N_t^-1 [(1 - lambda) R W + lambda 1_{I_t} (W^T qhat)^T]
                   over every row (dZ itself is never formed);
      SwiGLU:      dW_d = dy^T A, dA = dy W_d, dG = dA * U * SiLU'(G),
                   dU = dA * SiLU(G), dW_g = dG^T x, dW_u = dU^T x,
                   dx = dy + dG W_g + dU W_u;
      Linear(+GELU): dpre = dx (* GELU'(pre)), dW = dpre^T x, db = sum_i dpre_i,
                   dx = dpre W;
      RMSNorm:     dgamma = sum_i dy_i * xhat_i, dx = r (dy gamma - xhat
                   mean_j(dy_j gamma_j xhat_j)).
    Every cotangent is carried over all rows; a weight gradient is formed only
    on its sampled output rows.  rows[k] lists, for tensor k (interface order),
    the output rows of a matrix (row j of dW is column j of the layer's output
    cotangent contracted with its input) or the elements of a vector.  The
    input cotangent of the first layer is not needed and not formed.
    Returns one array per tensor: [len(rows[k]), cols] or [len(rows[k])]."""
    per_layer, (hw, hb) = _split_params(layers, head_bias, params)
    tape, h_last = saved
    R = np.asarray(R, dtype=F64)
    qhat = np.asarray(qhat, dtype=F64)
    vf = np.asarray(valid, dtype=F64)
    a, b = (1.0 - lam) / n_t, lam / n_t
    out: List[np.ndarray] = [None] * len(params)
    k = len(params) - 1
    if hb is not None:
        rb = np.asarray(rows[k])
        # sum_i dZ_ij = a sum_{i in I_t} r_ij + b N_t qhat_j (R is zero off I_t)
        out[k] = a * R[:, rb].sum(axis=0) + b * n_t * qhat[rb]
        k -= 1
    rw = np.asarray(rows[k])
    out[k] = (a * R[:, rw] + b * vf[:, None] * qhat[None, rw]).T @ h_last
    k -= 1
    hw = np.asarray(hw, dtype=F64)
    dx = a * (R @ hw) + b * vf[:, None] * (hw.T @ qhat)[None, :]
    for li in range(len(layers) - 1, -1, -1):
        kind = layers[li][0]
        rec = tape[li]
        below = li > 0
        if kind == "swiglu":
            wg, wu, wd = per_layer[li]
            _, x, G, U, A = rec
            dy = dx
            out[k] = dy[:, np.asarray(rows[k])].T @ A
            dA = dy @ wd
            dG = dA * U * silu_prime(G)
            dU = dA * silu(G)
            del dA
            out[k - 1] = dU[:, np.asarray(rows[k - 1])].T @ x
            out[k - 2] = dG[:, np.asarray(rows[k - 2])].T @ x
            k -= 3
            dx = dy + dG @ wg + dU @ wu if below else None
        elif kind == "rmsnorm":
            (gamma,) = per_layer[li]
            _, x, r, xhat = rec
            rg = np.asarray(rows[k])
            out[k] = (dx[:, rg] * xhat[:, rg]).sum(axis=0)
            k -= 1
            if below:
                dxhat = dx * gamma
                dx = r * (dxhat - xhat * np.mean(dxhat * xhat, axis=1, keepdims=True))
        else:
            w, bias = per_layer[li]
            _, x, pre = rec
            dpre = dx * gelu_prime(pre) if kind == "linear_gelu" else dx
            if bias is not None:
                out[k] = dpre[:, np.asarray(rows[k])].sum(axis=0)
                k -= 1
            out[k] = dpre[:, np.asarray(rows[k])].T @ x
            k -= 1
            dx = dpre @ w if below else None
    return out


# --------------------------------------------------------------------------
# Drift telemetry and the own-step control (Section 3.3, Eq. jacobian-drift
# and Eq. drift-telemetry; stale-control and drift-measurement appendices).
#
# The own-step control keeps BOM's task-space signal s_t but projects it
# through the model and examples of its own step, accumulating the
# parameter-shaped  M_t = beta1 M_{t-1} + (1 - beta1) Jbar_t^T s_t  and using
# u = (1 - lambda) g_t + lambda Mhat_t,  Mhat_t = M_t / (1 - beta1^t).
# On one trajectory, Mhat_t - h_t (h_t = Jbar_t^T qhat_t) is the
# bias-corrected historical-projection drift; the telemetry reports its cosine
# and relative size, and the within-batch cancellation ratio
# ||s_t|| / (N_t^-1 sum_{i in I_t} ||r_i||).
# --------------------------------------------------------------------------
def own_step_projection(layers, head_bias, params, X, labels, ignore_index=-100):
    """Jbar_t^T s_t per tensor: the reverse pass of the logit cotangent
    1_{I_t} s_t^T / N_t.  Returns (per-tensor list, s_t, N_t)."""
    params = [np.asarray(p, dtype=F64) for p in params]
    Z, saved = forward(layers, head_bias, params, X)
    valid, n_t = supervised_set(labels, Z.shape[1], ignore_index)
    s = batch_mean_residual(residuals(Z, labels, valid), n_t)
    o, _, _ = backward(layers, head_bias, params, saved, valid[:, None] * s[None, :] / n_t)
    return o, s, n_t


def own_step_moment(M_prev, o, t, beta1):
    """M_t = beta1 M_{t-1} + (1 - beta1) o_t and Mhat_t = M_t / (1 - beta1^t)
    (stale-control appendix; the bias correction as for q)."""
    if t < 1:
        raise OracleError("t is 1-based")
    M = beta1 * np.asarray(M_prev, dtype=F64) + (1.0 - beta1) * np.asarray(o, dtype=F64)
    return M, M / (1.0 - beta1 ** t)


def drift_statistics(mhat_list, h_list):
    """cos(Mhat, h) and ||Mhat - h|| / ||Mhat|| over the concatenation of the
    given tensors (Eq. drift-telemetry), with the four sums they come from."""
    a = np.concatenate([np.ravel(np.asarray(x, dtype=F64)) for x in mhat_list])
    b = np.concatenate([np.ravel(np.asarray(x, dtype=F64)) for x in h_list])
    dot, mm, hh = float(a @ b), float(a @ a), float(b @ b)
    dd = float((a - b) @ (a - b))
    return dict(dot=dot, mm=mm, hh=hh, dd=dd, cos=dot / math.sqrt(mm * hh), rel=math.sqrt(dd / mm))


def cancellation_ratio(R, valid, n_t):
    """||s_t|| / (N_t^-1 sum_{i in I_t} ||r_i||) (drift-measurement appendix:
    the share of the mean per-example residual norm that survives batch
    averaging).  Returns (ratio, ||s_t||, mean residual norm)."""
    rows = np.nonzero(valid)[0]
    s = R[rows].sum(axis=0) / n_t
    mean_norm = float(np.sqrt((R[rows] ** 2).sum(axis=1)).sum() / n_t)
    s_norm = float(np.sqrt(s @ s))
    return s_norm / mean_norm, s_norm, mean_norm


# --------------------------------------------------------------------------
# BOM-Adam-mini (Section 3.5 "The substitution", composition with Adam-mini;
# optimizer-implementation appendix): Adam-mini keeps one second-moment scalar
# per block of a tensor (per attention head, per output neuron, the whole
# tensor, or per element) and scales every element of the block by it.  The
# BOM composition feeds it u instead of a first moment:
#   v_b = beta2 v_b + (1 - beta2) mean_{i in b} u_i^2,   vhat_b = v_b / (1 - beta2^t)
#   theta_i <- (1 - eta omega) theta_i - eta u_i / (sqrt(vhat_b) + eps).
# Blocks here are consecutive runs of `block` elements of the flat tensor (a
# row-major [d_out, d_in] matrix with block = d_in shares v per output neuron;
# block = n is the whole tensor, block = 1 is elementwise BOM-AdamW); the last
# block may be shorter.
# --------------------------------------------------------------------------
def bom_update_blockshared(theta, u, v_blocks, block, lr, wd, t, beta2=0.999, eps=1e-8):
    """Returns (theta_new, v_blocks_new) in float64."""
    if t < 1:
        raise OracleError("t is 1-based")
    if block < 1:
        raise OracleError("block >= 1")
    theta = np.asarray(theta, dtype=F64).ravel()
    u = np.asarray(u, dtype=F64).ravel()
    n = theta.size
    nb = -(-n // block)
    v_blocks = np.asarray(v_blocks, dtype=F64).ravel()
    if v_blocks.size != nb:
        raise OracleError("one second-moment entry per block")
    mean_sq = np.array([np.mean(u[b * block:(b + 1) * block] ** 2) for b in range(nb)])
    v_new = beta2 * v_blocks + (1.0 - beta2) * mean_sq
    vhat = v_new / (1.0 - beta2 ** t)
    denom = np.repeat(np.sqrt(vhat) + eps, block)[:n]
    theta_new = (1.0 - lr * wd) * theta - lr * u / denom
    return theta_new, v_new


# --------------------------------------------------------------------------
# Global-norm clipping of the numerator (pretraining-parameters appendix: the
# language-modeling runs clip at 1.0; convergence appendix: the clipped
# numerator is what the adaptive update receives).  The norm runs over every
# trainable tensor together; the factor follows the common PyTorch rule
#   c = min(1, max_norm / (||u||_2 + 1e-6)),  u <- c u  before v and theta.
# --------------------------------------------------------------------------
def clip_factor(u_list, max_norm):
    """Scale applied to every tensor of u so that the global L2 norm is at most max_norm."""
    sq = sum(float(np.sum(np.asarray(u, dtype=F64) ** 2)) for u in u_list)
    return min(1.0, max_norm / (math.sqrt(sq) + 1e-6))


def bom_update_clipped(theta_list, u_list, v_list, lr, wd_list, t, max_norm, beta2=0.999, eps=1e-8):
    """BOM-AdamW update of several tensors with their numerator clipped to a
    global norm of max_norm.  Returns (theta_list, v_list, factor)."""
    c = clip_factor(u_list, max_norm)
    out_t, out_v = [], []
    for th, u, v, wd in zip(theta_list, u_list, v_list, wd_list):
        a, b = bom_update(th, c * np.asarray(u, dtype=F64), v, lr, wd, t, beta2, eps)
        out_t.append(a)
        out_v.append(b)
    return out_t, out_v, c
