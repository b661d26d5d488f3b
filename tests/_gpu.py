"""Helpers of the GPU parity tests: upload seeded inputs, run the C-ABI step and
update through the Python binding, and run the fp64 oracle on the same inputs."""
from __future__ import annotations

import numpy as np
import torch

import oracle as O
from paper_2609_36738_gb300 import bom as B
from paper_2609_36738_gb300 import inputs as I
from tests import _indep as X

DEV = "cuda"
TOL = {"f32": 1e-5, "bf16": 2e-2}


def ensure_built():
    from paper_2609_36738_gb300 import build
    build.build()
    B.lib()


def to_dev(arr: np.ndarray) -> torch.Tensor:
    if arr.dtype == np.uint16:
        return torch.from_numpy(np.ascontiguousarray(arr).view(np.int16)).to(DEV).view(torch.bfloat16)
    return torch.from_numpy(np.ascontiguousarray(arr)).to(DEV)


def np64(t: torch.Tensor) -> np.ndarray:
    return t.detach().float().cpu().double().numpy()


def host_f32(ptr: int, count: int) -> np.ndarray:
    return np.frombuffer(B.copy_to_host(ptr, 4 * count), dtype=np.float32).astype(np.float64)


rel_l2 = X.rel_l2


def bf16_round(a: np.ndarray) -> np.ndarray:
    """float64 values rounded to the nearest bf16 (through float32), as float64."""
    return I.bf16_to_f64(I.bf16_bits(np.asarray(a, dtype=np.float32)))


class GpuBom:
    """A handle plus device copies of a workload's parameters."""

    def __init__(self, wl: I.Workload, params_np, out_mode=B.BOM_OUT_U, lam=0.5, beta1=0.9, max_rows=None):
        self.wl = wl
        self.out_mode = out_mode
        self.model = B.BomModel(B.config_for(wl, lam, beta1, out_mode, max_rows))
        # numpy parameters are uploaded; device tensors are copied
        self.params = [p.clone() if isinstance(p, torch.Tensor) else to_dev(p) for p in params_np]
        self.q = torch.zeros(wl.vocab, dtype=torch.float32, device=DEV)

    def step(self, x_np, y_np, t, check=True):
        x = to_dev(x_np)
        y = torch.from_numpy(np.ascontiguousarray(y_np, dtype=np.int32)).to(DEV)
        grads = [torch.empty_like(p) for p in self.params]
        hs = None
        if self.out_mode == B.BOM_OUT_G_AND_H:
            hs = [torch.empty(p.shape, dtype=torch.float32, device=DEV) for p in self.params]
        self.model.step(x, y, x.shape[0], self.params, self.q, t, grads, hs)
        st = self.model.stats(check=check)
        qp, sp, lp = self.model.outputs()
        V = self.wl.vocab
        out = dict(stats=st, grads=grads, h=hs, q=np64(self.q))
        if st["code"] == B.BOM_OK:
            out["qhat"] = host_f32(qp, V)
            out["s"] = host_f32(sp, V)
            out["lse"] = host_f32(lp, x.shape[0])
        return out


def oracle_step(wl, params64, x_np, y_np, q_prev, t, lam=0.5, beta1=0.9):
    return O.bom_step(X.oracle_layers(wl), wl.head_bias, params64, X.x_f64(wl, x_np), y_np, q_prev, t,
                      lam=lam, beta1=beta1)


def weighted_step_check(th_gpu, th_in, th_ref, v_ref, t, beta2, tol):
    """Error and bound of an update step theta - theta_in (Section 3.4), each
    element weighed by its own sqrt(vhat) of the oracle: in that metric the
    step is about lr u, so its error is of the order of the error of u
    whatever the size of the element's own step (an element with tiny u still
    moves by about lr, and at t = 1 by -lr sign(u)).  The bound is tol times
    the weighted step, plus half an fp32 ulp of each updated element (the GPU
    stores theta in fp32: a step of lr = 1e-3 on theta near 1 is resolved to
    about 6e-5 of itself, whatever the accuracy of u).  Returns (err, bound)."""
    w = np.sqrt(np.asarray(v_ref, dtype=np.float64) / (1.0 - beta2 ** t))
    d = (np.asarray(th_gpu) - th_in) * w
    ref = (np.asarray(th_ref) - th_in) * w
    half_ulp = 0.5 * np.abs(np.spacing(np.asarray(th_ref, dtype=np.float32))).astype(np.float64)
    err = float(np.linalg.norm(d - ref))
    bound = tol * float(np.linalg.norm(ref)) + float(np.linalg.norm(half_ulp * w))
    return err, bound

