"""Python binding of ``libbom.so`` (argument marshalling only).

Every function mirrors the C entry point of the same name in ``include/bom.h``;
all computation happens in the library's CUDA kernels.  Tensor arguments may be
torch CUDA tensors (their ``data_ptr()`` is passed) or raw integer device
pointers.  ``stream=None`` means torch's current CUDA stream, so the library's
kernels are ordered with the caller's torch work.

Importing this module never falls back to anything: if the library is missing
or fails to load, :func:`lib` raises.
"""
from __future__ import annotations

import ctypes as C
import os
from typing import Optional, Sequence

from . import inputs as _inputs

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "_lib", "libbom.so")

(BOM_OK, BOM_EINVAL, BOM_ENOMEM, BOM_ECUDA, BOM_ELABEL, BOM_EEMPTY, BOM_ETIMEOUT, BOM_ENOTSUP, BOM_ENONFINITE,
 BOM_ESHARD) = range(10)
BOM_F32, BOM_BF16 = 0, 1
BOM_LAYER_LINEAR, BOM_LAYER_LINEAR_GELU, BOM_LAYER_SWIGLU, BOM_LAYER_RMSNORM = 0, 1, 2, 3
BOM_OUT_U, BOM_OUT_G_AND_H = 0, 1

# Every symbol include/bom.h declares.
EXPORTED = ("bom_param_count", "bom_param_shape", "bom_init", "bom_workspace_bytes", "bom_step",
            "bom_step_shard_begin", "bom_step_shard_end",
            "bom_step_vshard_begin", "bom_step_vshard_mid", "bom_step_vshard_end",
            "bom_set_input_grad", "bom_step_outputs", "bom_get_stats", "bom_get_stats_async", "bom_stats_decode",
            "bom_update", "bom_gemm_bf16", "bom_trace", "bom_trace_read",
            "bom_launch_count", "bom_colsum_noalloc", "bom_set_own_step_output", "bom_own_step_moment",
            "bom_stats_transfer_bytes", "bom_update_blockshared", "bom_sqnorm", "bom_update_clipped",
            "bom_set_fused_update", "bom_set_step_scalars", "bom_graph_capture", "bom_graph_launch",
            "bom_graph_destroy", "bom_destroy", "bom_status_string")


class bom_trace_entry(C.Structure):
    _fields_ = [("name", C.c_char_p), ("flops", C.c_double), ("bytes", C.c_double), ("ms", C.c_float)]


class bom_layer(C.Structure):
    _fields_ = [("kind", C.c_int32), ("has_bias", C.c_int32), ("d_in", C.c_int64), ("d_out", C.c_int64)]


class bom_config(C.Structure):
    _fields_ = [("max_rows", C.c_int64), ("d_in", C.c_int64), ("d_out", C.c_int64), ("n_layers", C.c_int32),
                ("layers", C.POINTER(bom_layer)), ("head_bias", C.c_int32), ("compute", C.c_int32),
                ("lambda_", C.c_float), ("beta1", C.c_float), ("ignore_index", C.c_int32),
                ("out_mode", C.c_int32)]


class bom_stats(C.Structure):
    _fields_ = [("loss", C.c_float), ("n_t", C.c_int32), ("status", C.c_int32), ("s_norm", C.c_float),
                ("r_norm_mean", C.c_float), ("cancel", C.c_float)]


class BomError(RuntimeError):
    def __init__(self, code: int, where: str):
        self.code = code
        super().__init__(f"{where}: {status_string(code)}")


_LIB = None


def lib() -> C.CDLL:
    """Loads libbom.so; raises if it has not been built."""
    global _LIB
    if _LIB is not None:
        return _LIB
    if not os.path.exists(LIB_PATH):
        raise RuntimeError(f"{LIB_PATH} is missing: build it with paper_2609_36738_gb300.build.build()")
    L = C.CDLL(LIB_PATH)
    vp, i64, i32, f32 = C.c_void_p, C.c_int64, C.c_int32, C.c_float
    L.bom_param_count.argtypes = [C.POINTER(bom_config)]
    L.bom_param_count.restype = i32
    L.bom_param_shape.argtypes = [C.POINTER(bom_config), i32, C.POINTER(i64), C.POINTER(i64)]
    L.bom_param_shape.restype = i32
    L.bom_init.argtypes = [C.POINTER(vp), C.POINTER(bom_config)]
    L.bom_init.restype = i32
    L.bom_workspace_bytes.argtypes = [C.POINTER(bom_config)]
    L.bom_workspace_bytes.restype = i64
    L.bom_step.argtypes = [vp, vp, vp, i64, C.POINTER(vp), vp, i64, C.POINTER(vp), C.POINTER(vp), vp]
    L.bom_step.restype = i32
    L.bom_step_shard_begin.argtypes = [vp, vp, vp, i64, C.POINTER(vp), vp, vp]
    L.bom_step_shard_begin.restype = i32
    L.bom_step_shard_end.argtypes = [vp, vp, vp, i64, C.POINTER(vp), vp, i64, vp, C.POINTER(vp), C.POINTER(vp), vp]
    L.bom_step_shard_end.restype = i32
    L.bom_step_vshard_begin.argtypes = [vp, vp, vp, i64, C.POINTER(vp), i64, i64, vp, vp]
    L.bom_step_vshard_begin.restype = i32
    L.bom_step_vshard_mid.argtypes = [vp, vp, vp, i64, C.POINTER(vp), vp, i64, vp, i32, C.POINTER(vp), vp, vp]
    L.bom_step_vshard_mid.restype = i32
    L.bom_step_vshard_end.argtypes = [vp, vp, vp, i64, C.POINTER(vp), vp, C.POINTER(vp), vp]
    L.bom_step_vshard_end.restype = i32
    L.bom_set_input_grad.argtypes = [vp, vp]
    L.bom_set_input_grad.restype = i32
    L.bom_step_outputs.argtypes = [vp, C.POINTER(vp), C.POINTER(vp), C.POINTER(vp)]
    L.bom_step_outputs.restype = i32
    L.bom_get_stats.argtypes = [vp, C.POINTER(bom_stats), vp]
    L.bom_get_stats.restype = i32
    L.bom_get_stats_async.argtypes = [vp, vp, vp]
    L.bom_get_stats_async.restype = i32
    L.bom_stats_decode.argtypes = [vp, C.POINTER(bom_stats)]
    L.bom_stats_decode.restype = i32
    L.bom_update.argtypes = [vp, vp, i32, vp, vp, vp, i64, f32, f32, f32, f32, f32, i64, vp]
    L.bom_update.restype = i32
    L.bom_gemm_bf16.argtypes = [vp, i64, i32, vp, i64, i32, vp, i64, i64, i64, i64, f32, vp]
    L.bom_gemm_bf16.restype = i32
    L.bom_trace.argtypes = [vp, i32]
    L.bom_trace.restype = i32
    L.bom_trace_read.argtypes = [vp, C.POINTER(bom_trace_entry), i32, vp]
    L.bom_trace_read.restype = i32
    L.bom_launch_count.argtypes = []
    L.bom_launch_count.restype = i64
    L.bom_colsum_noalloc.argtypes = [vp, i32, i64, i64, i64, vp, vp, vp]
    L.bom_colsum_noalloc.restype = i32
    L.bom_set_own_step_output.argtypes = [vp, C.POINTER(vp)]
    L.bom_set_own_step_output.restype = i32
    L.bom_own_step_moment.argtypes = [vp, vp, vp, vp, vp, i64, f32, i64, vp, vp]
    L.bom_own_step_moment.restype = i32
    L.bom_stats_transfer_bytes.argtypes = []
    L.bom_stats_transfer_bytes.restype = i64
    L.bom_update_blockshared.argtypes = [vp, vp, i32, vp, vp, vp, i64, i64, f32, f32, f32, f32, f32, i64, vp]
    L.bom_update_blockshared.restype = i32
    L.bom_sqnorm.argtypes = [vp, vp, i32, vp, f32, i64, vp, vp]
    L.bom_sqnorm.restype = i32
    L.bom_update_clipped.argtypes = [vp, vp, i32, vp, vp, vp, i64, f32, f32, f32, f32, f32, i64, vp, f32, vp]
    L.bom_update_clipped.restype = i32
    L.bom_set_fused_update.argtypes = [vp, C.POINTER(vp), C.POINTER(vp), C.POINTER(f32), f32, f32, f32]
    L.bom_set_fused_update.restype = i32
    L.bom_set_step_scalars.argtypes = [vp, vp, vp]
    L.bom_set_step_scalars.restype = i32
    L.bom_graph_capture.argtypes = [vp, vp, vp, i64, C.POINTER(vp), vp, C.POINTER(vp), C.POINTER(vp),
                                    C.POINTER(vp)]
    L.bom_graph_capture.restype = i32
    L.bom_graph_launch.argtypes = [vp, vp]
    L.bom_graph_launch.restype = i32
    L.bom_graph_destroy.argtypes = [vp]
    L.bom_graph_destroy.restype = None
    L.bom_destroy.argtypes = [vp]
    L.bom_destroy.restype = None
    L.bom_status_string.argtypes = [i32]
    L.bom_status_string.restype = C.c_char_p
    _LIB = L
    return L


def status_string(code: int) -> str:
    return lib().bom_status_string(int(code)).decode()


def _ptr(t) -> Optional[int]:
    if t is None:
        return None
    if isinstance(t, int):
        return t
    return t.data_ptr()


def _stream(stream) -> Optional[int]:
    if stream is None:
        import torch
        return torch.cuda.current_stream().cuda_stream
    if isinstance(stream, int):
        return stream
    return stream.cuda_stream


def _check(code: int, where: str):
    if code != BOM_OK:
        raise BomError(code, where)


# ---------------------------------------------------------------- config helpers
def make_config(max_rows: int, d_in: int, d_out: int, layers: Sequence, head_bias: bool, compute: int,
                lam: float = 0.5, beta1: float = 0.9, ignore_index: int = -100, out_mode: int = BOM_OUT_U):
    """bom_config from plain values; ``layers`` is a sequence of (kind, has_bias, d_in, d_out)."""
    arr = (bom_layer * max(len(layers), 1))()
    for i, (k, b, di, do) in enumerate(layers):
        arr[i] = bom_layer(int(k), int(b), int(di), int(do))
    cfg = bom_config(int(max_rows), int(d_in), int(d_out), len(layers), arr, int(head_bias), int(compute),
                     float(lam), float(beta1), int(ignore_index), int(out_mode))
    cfg._keep = arr  # keep the layer array alive with the struct
    return cfg


_KIND = {_inputs.LINEAR: BOM_LAYER_LINEAR, _inputs.LINEAR_GELU: BOM_LAYER_LINEAR_GELU,
         _inputs.SWIGLU: BOM_LAYER_SWIGLU, _inputs.RMSNORM: BOM_LAYER_RMSNORM}


def config_for(wl: "_inputs.Workload", lam: float = 0.5, beta1: float = 0.9, out_mode: int = BOM_OUT_U,
               max_rows: Optional[int] = None):
    layers = [(_KIND[l.kind], l.has_bias, l.d_in, l.d_out) for l in wl.layers]
    return make_config(max_rows or wl.n_rows, wl.d_in, wl.vocab, layers, wl.head_bias,
                       BOM_BF16 if wl.dtype == "bf16" else BOM_F32, lam, beta1, _inputs.IGNORE_INDEX, out_mode)


# ---------------------------------------------------------------- entry points
def bom_param_count(cfg: bom_config) -> int:
    return int(lib().bom_param_count(C.byref(cfg)))


def bom_param_shape(cfg: bom_config, index: int):
    r, c = C.c_int64(), C.c_int64()
    _check(lib().bom_param_shape(C.byref(cfg), int(index), C.byref(r), C.byref(c)), "bom_param_shape")
    return (r.value,) if c.value == 0 else (r.value, c.value)


def bom_workspace_bytes(cfg: bom_config) -> int:
    return int(lib().bom_workspace_bytes(C.byref(cfg)))


def bom_init(cfg: bom_config) -> C.c_void_p:
    h = C.c_void_p()
    _check(lib().bom_init(C.byref(h), C.byref(cfg)), "bom_init")
    return h


def bom_destroy(h) -> None:
    if h:
        lib().bom_destroy(h)


def bom_step(h, x, labels, n_rows: int, params, q, t: int, grads, h_out=None, stream=None) -> None:
    n = len(params)
    P = (C.c_void_p * n)(*[_ptr(p) for p in params])
    G = (C.c_void_p * n)(*[_ptr(g) for g in grads]) if grads is not None else None
    H = (C.c_void_p * n)(*[_ptr(p) for p in h_out]) if h_out is not None else None
    _check(lib().bom_step(h, _ptr(x), _ptr(labels), int(n_rows), P, _ptr(q), int(t), G,
                          H if H is not None else None, _stream(stream)), "bom_step")


def bom_step_shard_begin(h, x, labels, n_rows: int, params, xch, stream=None) -> None:
    n = len(params)
    P = (C.c_void_p * n)(*[_ptr(p) for p in params])
    _check(lib().bom_step_shard_begin(h, _ptr(x), _ptr(labels), int(n_rows), P, _ptr(xch), _stream(stream)),
           "bom_step_shard_begin")


def bom_step_shard_end(h, x, labels, n_rows: int, params, q, t: int, xch, grads, h_out=None, stream=None) -> None:
    n = len(params)
    P = (C.c_void_p * n)(*[_ptr(p) for p in params])
    G = (C.c_void_p * n)(*[_ptr(g) for g in grads]) if grads is not None else None
    H = (C.c_void_p * n)(*[_ptr(p) for p in h_out]) if h_out is not None else None
    _check(lib().bom_step_shard_end(h, _ptr(x), _ptr(labels), int(n_rows), P, _ptr(q), int(t), _ptr(xch), G, H,
                                    _stream(stream)), "bom_step_shard_end")


def bom_step_vshard_begin(h, x, labels, n_rows: int, params, v_total: int, v_first: int, lse_part,
                          stream=None) -> None:
    n = len(params)
    P = (C.c_void_p * n)(*[_ptr(p) for p in params])
    _check(lib().bom_step_vshard_begin(h, _ptr(x), _ptr(labels), int(n_rows), P, int(v_total), int(v_first),
                                       _ptr(lse_part), _stream(stream)), "bom_step_vshard_begin")


def bom_step_vshard_mid(h, x, labels, n_rows: int, params, q, t: int, lse_parts, n_shards: int, grads,
                        dh_part=None, stream=None) -> None:
    n = len(params)
    P = (C.c_void_p * n)(*[_ptr(p) for p in params])
    G = (C.c_void_p * n)(*[_ptr(g) for g in grads]) if grads is not None else None
    _check(lib().bom_step_vshard_mid(h, _ptr(x), _ptr(labels), int(n_rows), P, _ptr(q), int(t), _ptr(lse_parts),
                                     int(n_shards), G, _ptr(dh_part), _stream(stream)), "bom_step_vshard_mid")


def bom_step_vshard_end(h, x, labels, n_rows: int, params, dh_sum, grads, stream=None) -> None:
    n = len(params)
    P = (C.c_void_p * n)(*[_ptr(p) for p in params])
    G = (C.c_void_p * n)(*[_ptr(g) for g in grads]) if grads is not None else None
    _check(lib().bom_step_vshard_end(h, _ptr(x), _ptr(labels), int(n_rows), P, _ptr(dh_sum), G, _stream(stream)),
           "bom_step_vshard_end")


def bom_set_step_scalars(h, t_dev, lr_dev=None) -> None:
    """Registers the device step counter (int64) and, optionally, the device
    learning rate (fp32) that bom_step reads instead of its host values."""
    _check(lib().bom_set_step_scalars(h, _ptr(t_dev), _ptr(lr_dev)), "bom_set_step_scalars")


def bom_graph_capture(h, x, labels, n_rows: int, params, q, grads, h_out=None) -> C.c_void_p:
    n = len(params)
    P = (C.c_void_p * n)(*[_ptr(p) for p in params])
    G = (C.c_void_p * n)(*[_ptr(g) for g in grads]) if grads is not None else None
    H = (C.c_void_p * n)(*[_ptr(p) for p in h_out]) if h_out is not None else None
    g = C.c_void_p()
    _check(lib().bom_graph_capture(h, _ptr(x), _ptr(labels), int(n_rows), P, _ptr(q), G, H, C.byref(g)),
           "bom_graph_capture")
    return g


def bom_graph_launch(g, stream=None) -> None:
    _check(lib().bom_graph_launch(g, _stream(stream)), "bom_graph_launch")


def bom_graph_destroy(g) -> None:
    if g:
        lib().bom_graph_destroy(g)


def bom_set_input_grad(h, dx) -> None:
    _check(lib().bom_set_input_grad(h, _ptr(dx)), "bom_set_input_grad")


def bom_step_outputs(h):
    q, s, l = C.c_void_p(), C.c_void_p(), C.c_void_p()
    _check(lib().bom_step_outputs(h, C.byref(q), C.byref(s), C.byref(l)), "bom_step_outputs")
    return q.value, s.value, l.value


def bom_get_stats(h, stream=None, check: bool = True) -> dict:
    st = bom_stats()
    code = lib().bom_get_stats(h, C.byref(st), _stream(stream))
    if check:
        _check(code, "bom_get_stats")
    return dict(loss=st.loss, n_t=st.n_t, status=st.status, s_norm=st.s_norm, r_norm_mean=st.r_norm_mean,
                cancel=st.cancel, code=code)


def bom_get_stats_async(h, dst, stream=None) -> None:
    """Enqueue the copy of the last step's statistics block into host memory
    ``dst`` (a pinned uint8 tensor of bom_stats_transfer_bytes() bytes)."""
    _check(lib().bom_get_stats_async(h, _ptr(dst), _stream(stream)), "bom_get_stats_async")


def bom_stats_decode(src, check: bool = True) -> dict:
    """The statistics held in ``src`` (filled by bom_get_stats_async)."""
    st = bom_stats()
    code = lib().bom_stats_decode(_ptr(src), C.byref(st))
    if check:
        _check(code, "bom_stats_decode")
    return dict(loss=st.loss, n_t=st.n_t, status=st.status, s_norm=st.s_norm, r_norm_mean=st.r_norm_mean,
                cancel=st.cancel, code=code)


def bom_update(theta, g, g_dtype: int, hvec, v, theta_bf16, n: int, lr: float, wd: float, lam: float,
               beta2: float, eps: float, t: int, stream=None) -> None:
    _check(lib().bom_update(_ptr(theta), _ptr(g), int(g_dtype), _ptr(hvec), _ptr(v), _ptr(theta_bf16), int(n),
                            float(lr), float(wd), float(lam), float(beta2), float(eps), int(t), _stream(stream)),
           "bom_update")


def bom_set_fused_update(h, theta, v, wd, lr: float, beta2: float, eps: float) -> None:
    """Registers per-tensor fp32 master weights, second moments and weight
    decays for the update fused into bom_step (``theta=None`` disables it)."""
    if theta is None:
        _check(lib().bom_set_fused_update(h, None, None, None, 0.0, 0.0, 0.0), "bom_set_fused_update")
        return
    n = len(theta)
    T = (C.c_void_p * n)(*[_ptr(p) for p in theta])
    Vv = (C.c_void_p * n)(*[_ptr(p) for p in v])
    W = (C.c_float * n)(*[float(w) for w in wd])
    _check(lib().bom_set_fused_update(h, T, Vv, W, float(lr), float(beta2), float(eps)), "bom_set_fused_update")


def bom_update_blockshared(theta, g, g_dtype: int, hvec, v_blocks, theta_bf16, n: int, block: int, lr: float,
                           wd: float, lam: float, beta2: float, eps: float, t: int, stream=None) -> None:
    _check(lib().bom_update_blockshared(_ptr(theta), _ptr(g), int(g_dtype), _ptr(hvec), _ptr(v_blocks),
                                        _ptr(theta_bf16), int(n), int(block), float(lr), float(wd), float(lam),
                                        float(beta2), float(eps), int(t), _stream(stream)), "bom_update_blockshared")


def bom_sqnorm(h, g, g_dtype: int, hvec, lam: float, n: int, sq, stream=None) -> None:
    _check(lib().bom_sqnorm(h, _ptr(g), int(g_dtype), _ptr(hvec), float(lam), int(n), _ptr(sq), _stream(stream)),
           "bom_sqnorm")


def bom_update_clipped(theta, g, g_dtype: int, hvec, v, theta_bf16, n: int, lr: float, wd: float, lam: float,
                       beta2: float, eps: float, t: int, sq, max_norm: float, stream=None) -> None:
    _check(lib().bom_update_clipped(_ptr(theta), _ptr(g), int(g_dtype), _ptr(hvec), _ptr(v), _ptr(theta_bf16), int(n),
                                    float(lr), float(wd), float(lam), float(beta2), float(eps), int(t), _ptr(sq),
                                    float(max_norm), _stream(stream)), "bom_update_clipped")


def bom_gemm_bf16(A, lda: int, a_mn_major: bool, B, ldb: int, b_mn_major: bool, D, ldd: int, M: int, N: int,
                  K: int, alpha: float = 1.0, stream=None) -> None:
    _check(lib().bom_gemm_bf16(_ptr(A), int(lda), int(a_mn_major), _ptr(B), int(ldb), int(b_mn_major), _ptr(D),
                               int(ldd), int(M), int(N), int(K), float(alpha), _stream(stream)), "bom_gemm_bf16")


def bom_trace(h, enable: bool) -> None:
    _check(lib().bom_trace(h, int(bool(enable))), "bom_trace")


def bom_trace_read(h, stream=None, max_entries: int = 256):
    """[(name, flops, bytes, ms)] for every launch of the last traced step."""
    buf = (bom_trace_entry * max_entries)()
    n = lib().bom_trace_read(h, buf, max_entries, _stream(stream))
    if n < 0:
        raise BomError(BOM_ECUDA, "bom_trace_read")
    return [(buf[i].name.decode(), buf[i].flops, buf[i].bytes, buf[i].ms) for i in range(min(n, max_entries))]


def bom_launch_count() -> int:
    return int(lib().bom_launch_count())


def bom_colsum_noalloc(x, dtype: int, ldx: int, n_rows: int, n_cols: int, weights, out, stream=None) -> None:
    """out[j] = sum_i w_i x[i, j] without any device allocation (fixed 4 MiB
    scratch inside the library; see include/bom.h for the limits)."""
    _check(lib().bom_colsum_noalloc(_ptr(x), int(dtype), int(ldx), int(n_rows), int(n_cols), _ptr(weights),
                                    _ptr(out), _stream(stream)), "bom_colsum_noalloc")


def bom_set_own_step_output(h, o) -> None:
    """Registers per-tensor fp32 outputs of the own-step projection Jbar^T s_t
    (``None`` disables it)."""
    if o is None:
        _check(lib().bom_set_own_step_output(h, None), "bom_set_own_step_output")
        return
    O = (C.c_void_p * len(o))(*[_ptr(p) for p in o])
    _check(lib().bom_set_own_step_output(h, O), "bom_set_own_step_output")


def bom_own_step_moment(h, M, o, hvec, mhat, n: int, beta1: float, t: int, sums=None, stream=None) -> None:
    _check(lib().bom_own_step_moment(h, _ptr(M), _ptr(o), _ptr(hvec), _ptr(mhat), int(n), float(beta1), int(t),
                                     _ptr(sums), _stream(stream)), "bom_own_step_moment")


def bom_stats_transfer_bytes() -> int:
    return int(lib().bom_stats_transfer_bytes())


class BomModel:
    """Owns a handle for one configuration (RAII around bom_init / bom_destroy)."""

    def __init__(self, cfg: bom_config):
        self.cfg = cfg
        self.h = bom_init(cfg)
        self.n_params = bom_param_count(cfg)
        self.shapes = [bom_param_shape(cfg, i) for i in range(self.n_params)]

    def step(self, x, labels, n_rows, params, q, t, grads, h_out=None, stream=None):
        bom_step(self.h, x, labels, n_rows, params, q, t, grads, h_out, stream)

    def stats(self, stream=None, check=True):
        return bom_get_stats(self.h, stream, check)

    def outputs(self):
        return bom_step_outputs(self.h)

    def close(self):
        if self.h:
            bom_destroy(self.h)
            self.h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass


# ---------------------------------------------------------------- device copies
_CUDART = None


def copy_to_host(ptr: int, nbytes: int) -> bytes:
    """cudaMemcpy of ``nbytes`` from device pointer ``ptr`` (library workspace
    outputs such as bom_step_outputs) into a host buffer."""
    global _CUDART
    lib()
    if _CUDART is None:
        _CUDART = C.CDLL("libcudart.so.13")
        _CUDART.cudaMemcpy.argtypes = [C.c_void_p, C.c_void_p, C.c_size_t, C.c_int]
        _CUDART.cudaMemcpy.restype = C.c_int
    buf = C.create_string_buffer(int(nbytes))
    rc = _CUDART.cudaMemcpy(buf, C.c_void_p(ptr), C.c_size_t(int(nbytes)), 2)
    if rc != 0:
        raise RuntimeError(f"cudaMemcpy failed with {rc}")
    return buf.raw
