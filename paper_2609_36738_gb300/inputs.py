"""Seeded synthetic workloads for the BOM task-space momentum pass.

This module only *generates data*: model shapes, parameter initialisations,
batches of inputs and labels, and the flat buffers of the update sweep.  It
holds none of the method's arithmetic (no softmax, no residual, no EMA, no
gradient, no update rule), so that the fp64 oracle under ``oracle/`` and the
CUDA path can both be fed from it without sharing any computation.

Every tensor comes from ``numpy.random.default_rng([seed, tag])`` (PCG64), so
the same seed yields the same bytes on x86 and on Arm.  bf16 tensors are
returned as their raw ``uint16`` bit patterns (round-to-nearest-even from the
float32 draw); the float value each side computes with is exactly the value
those bits encode.

Workloads (shapes follow the paper's settings; the data are synthetic because
the paper's corpora and datasets are not available here):

* ``tiny_mlp_f32``     64 -> 128 (GELU) -> 10 classes, batch 32, fp32
  (the STL10-like classification setting of Table cost-model, B*C = 320).
* ``vision_head_bf16`` 768 -> 3072 -> 768 (GELU after each) -> 1000 classes,
  batch 256, bf16 (ImageNet-like output space, B = 256, C = 1000).
* ``lm_head_bf16``     hidden states 8192 x 768, head 50257 x 768, Zipf(1.1)
  next-token labels (the vocabulary-space construction of the LM appendix).
* ``lm_mlp_bf16``      two SwiGLU MLP sublayers (d = 2048, ffn = 8192) under a
  32000-token head, 16384 tokens, Zipf(1.1) labels.
* update sweep         flat fp32 theta / fp32 h / fp32 v and bf16 g buffers.

Small variants with the same structure and ragged sizes serve the parity
tests.
"""
from __future__ import annotations

import dataclasses
from typing import List, Optional, Sequence, Tuple

import numpy as np

IGNORE_INDEX = -100

# Layer kinds of the backbone, in the order the C interface numbers them.
LINEAR = "linear"
LINEAR_GELU = "linear_gelu"
SWIGLU = "swiglu"
RMSNORM = "rmsnorm"


# --------------------------------------------------------------------------
# bf16 storage helpers (bit-level data marshalling only)
# --------------------------------------------------------------------------
def bf16_bits(x: np.ndarray) -> np.ndarray:
    """Round float32 values to bf16 (nearest, ties to even); return uint16 bits."""
    f = np.ascontiguousarray(x, dtype=np.float32)
    u = f.view(np.uint32).astype(np.uint64)
    nan = np.isnan(f)
    rounded = (u + 0x7FFF + ((u >> 16) & 1)) >> 16
    out = rounded.astype(np.uint16)
    out[nan] = 0x7FC0
    return out


def bf16_to_f32(bits: np.ndarray) -> np.ndarray:
    """Expand uint16 bf16 bit patterns to the float32 values they encode."""
    b = np.ascontiguousarray(bits, dtype=np.uint16)
    return (b.astype(np.uint32) << 16).view(np.float32)


def bf16_to_f64(bits: np.ndarray) -> np.ndarray:
    return bf16_to_f32(bits).astype(np.float64)


# --------------------------------------------------------------------------
# Model / workload description
# --------------------------------------------------------------------------
@dataclasses.dataclass(frozen=True)
class Layer:
    kind: str          # LINEAR, LINEAR_GELU, SWIGLU or RMSNORM (d_out = d_in)
    d_in: int          # input width (d_model for SWIGLU)
    d_out: int         # output width (ffn width for SWIGLU; output stays d_model)
    has_bias: bool = False


@dataclasses.dataclass(frozen=True)
class Workload:
    name: str
    n_rows: int                  # supervised rows per batch (examples / tokens)
    d_in: int                    # width of the input X
    layers: Tuple[Layer, ...]    # backbone, applied in order
    vocab: int                   # d_out of the head (classes / vocabulary)
    head_bias: bool
    dtype: str                   # "f32" or "bf16"
    labels: str                  # "uniform" or "zipf"
    steps: int = 1
    head_init: str = "kaiming"   # "kaiming" or "normal002"
    ignore_frac: float = 0.0     # fraction of rows whose label is IGNORE_INDEX

    @property
    def d_model(self) -> int:
        w = self.d_in
        for l in self.layers:
            w = l.d_in if l.kind == SWIGLU else l.d_out
        return w

    def param_shapes(self) -> List[Tuple[str, Tuple[int, ...], bool]]:
        """(name, shape, is_matrix) of every trainable tensor, in interface order."""
        out = []
        w = self.d_in
        for li, l in enumerate(self.layers):
            if l.kind == SWIGLU:
                assert l.d_in == w
                out.append((f"l{li}.w_gate", (l.d_out, l.d_in), True))
                out.append((f"l{li}.w_up", (l.d_out, l.d_in), True))
                out.append((f"l{li}.w_down", (l.d_in, l.d_out), True))
            elif l.kind == RMSNORM:
                assert l.d_in == w and l.d_out == w
                out.append((f"l{li}.norm_weight", (w,), False))
            else:
                assert l.d_in == w
                out.append((f"l{li}.weight", (l.d_out, l.d_in), True))
                if l.has_bias:
                    out.append((f"l{li}.bias", (l.d_out,), False))
                w = l.d_out
        out.append(("head.weight", (self.vocab, w), True))
        if self.head_bias:
            out.append(("head.bias", (self.vocab,), False))
        return out

    def n_params(self) -> int:
        return int(sum(int(np.prod(s)) for _, s, _ in self.param_shapes()))


def _rng(seed: int, *tag: int) -> np.random.Generator:
    return np.random.default_rng([int(seed) & 0xFFFFFFFF, *[int(t) for t in tag]])


def _store(x32: np.ndarray, dtype: str) -> np.ndarray:
    return bf16_bits(x32) if dtype == "bf16" else np.ascontiguousarray(x32, dtype=np.float32)


def init_params(wl: Workload, seed: int = 0) -> List[np.ndarray]:
    """Initial parameters in storage form (float32, or bf16 bits as uint16).

    Matrices: Kaiming-uniform U(-sqrt(6/fan_in), +sqrt(6/fan_in)); the LM head
    uses N(0, 0.02) when ``head_init == "normal002"``.  Biases start at zero.
    RMSNorm weights are 1 + N(0, 0.1^2) (not all ones, so that the weight's
    own gradient path carries signal in the checks).
    """
    out = []
    for k, (name, shape, is_mat) in enumerate(wl.param_shapes()):
        g = _rng(seed, 1000 + k)
        if name.endswith("norm_weight"):
            x = (1.0 + 0.1 * g.standard_normal(shape)).astype(np.float32)
        elif not is_mat:
            x = np.zeros(shape, dtype=np.float32)
        elif name == "head.weight" and wl.head_init == "normal002":
            x = (g.standard_normal(shape, dtype=np.float32) * np.float32(0.02))
        else:
            bound = np.float32(np.sqrt(6.0 / shape[1]))
            x = g.uniform(-1.0, 1.0, size=shape).astype(np.float32) * bound
        out.append(_store(x, wl.dtype))
    return out


def zipf_labels(g: np.random.Generator, n: int, vocab: int, a: float = 1.1) -> np.ndarray:
    """Zipf(a) over ranks 1..vocab (truncated), rank k -> token id k-1 (inverse CDF)."""
    ranks = np.arange(1, vocab + 1, dtype=np.float64)
    w = ranks ** (-a)
    cdf = np.cumsum(w)
    cdf /= cdf[-1]
    u = g.random(n)
    idx = np.searchsorted(cdf, u, side="right")
    return np.minimum(idx, vocab - 1).astype(np.int32)


def make_batch(wl: Workload, seed: int = 0, step: int = 1) -> Tuple[np.ndarray, np.ndarray]:
    """(X, labels) for optimizer step ``step`` (1-based).  X is N(0,1)."""
    g = _rng(seed, 2000 + step)
    x = g.standard_normal((wl.n_rows, wl.d_in), dtype=np.float32)
    if wl.labels == "zipf":
        y = zipf_labels(g, wl.n_rows, wl.vocab)
    else:
        y = g.integers(0, wl.vocab, size=wl.n_rows, dtype=np.int64).astype(np.int32)
    if wl.ignore_frac > 0:
        drop = g.random(wl.n_rows) < wl.ignore_frac
        y[drop] = IGNORE_INDEX
    return _store(x, wl.dtype), y


def weight_decay_mask(wl: Workload, omega: float) -> List[float]:
    """Decoupled weight-decay coefficient per tensor: omega for matrices, 0 for
    biases and normalisation weights."""
    return [omega if is_mat else 0.0 for _, _, is_mat in wl.param_shapes()]


# --------------------------------------------------------------------------
# Named workloads
# --------------------------------------------------------------------------
TINY_MLP_F32 = Workload("tiny_mlp_f32", 32, 64, (Layer(LINEAR_GELU, 64, 128, True),),
                        10, True, "f32", "uniform", steps=5)
VISION_HEAD_BF16 = Workload("vision_head_bf16", 256, 768,
                            (Layer(LINEAR_GELU, 768, 3072, True), Layer(LINEAR_GELU, 3072, 768, True)),
                            1000, True, "bf16", "uniform", steps=20)
LM_HEAD_BF16 = Workload("lm_head_bf16", 8192, 768, (), 50257, False, "bf16", "zipf",
                        head_init="normal002")
LM_MLP_BF16 = Workload("lm_mlp_bf16", 16384, 2048,
                       (Layer(SWIGLU, 2048, 8192), Layer(SWIGLU, 2048, 8192)),
                       32000, False, "bf16", "zipf", head_init="normal002")
UPDATE_SIZES = (10_000_000, 125_000_000, 1_000_000_000)

# Small variants: same structure, ragged sizes (not multiples of the tiles).
LM_HEAD_SMALL = Workload("lm_head_small", 300, 136, (), 1003, False, "bf16", "zipf",
                         head_init="normal002", ignore_frac=0.1)
LM_MLP_SMALL = Workload("lm_mlp_small", 260, 128,
                        (Layer(SWIGLU, 128, 320), Layer(SWIGLU, 128, 320)),
                        777, False, "bf16", "zipf", head_init="normal002", ignore_frac=0.05)
VISION_SMALL = Workload("vision_small", 70, 96,
                        (Layer(LINEAR_GELU, 96, 200, True), Layer(LINEAR_GELU, 200, 88, True)),
                        130, True, "bf16", "uniform", steps=3)
# More than 128 rows (ragged: 300) with biased GELU layers: with the update
# registered, each layer's bias gradient comes from the column sums that the
# GEMM writing its output cotangent forms per 32-row block.
VISION_MID = Workload("vision_mid", 300, 96,
                      (Layer(LINEAR_GELU, 96, 200, True), Layer(LINEAR_GELU, 200, 88, True)),
                      130, True, "bf16", "uniform", steps=3)
# A tiny bf16 classifier (48 rows, 26 classes): its task-space pass runs in
# one CTA from shared memory, as the fp32 tiny ones do.
TINY_BF16 = Workload("tiny_bf16", 48, 64, (Layer(LINEAR_GELU, 64, 96, True),), 26, True, "bf16", "uniform",
                     steps=3, ignore_frac=0.1)
# A batch of 1000 rows with a 1536-wide GELU layer: its first forward layer
# and the second layer's input cotangent have enough tiles for CTA-pair
# 256 x 256 tiles (bias + GELU, and GELU' epilogues on that path), ragged in
# rows; with the update registered, that cotangent GEMM also forms the first
# layer's bias column sums per 32-row block on the pair tiles.
VISION_WIDE = Workload("vision_wide", 1000, 256,
                       (Layer(LINEAR_GELU, 256, 1536, True), Layer(LINEAR_GELU, 1536, 256, True)),
                       500, True, "bf16", "uniform", steps=2, ignore_frac=0.05)
TINY_RAGGED_F32 = Workload("tiny_ragged_f32", 37, 29, (Layer(LINEAR_GELU, 29, 45, True),
                                                       Layer(LINEAR, 45, 33, True)),
                           7, True, "f32", "uniform", steps=3, ignore_frac=0.1)

# Few output tiles and a long contraction in the head's input-side backward
# (256 rows x 128 columns, K = 8192): exercises the split-K path of the GEMMs.
LM_HEAD_WIDE = Workload("lm_head_wide", 256, 128, (), 8192, False, "bf16", "zipf",
                        head_init="normal002", ignore_frac=0.05)

# SwiGLU widths above one 128-row tile everywhere (d 256, ffn 576), so the
# three weight-gradient GEMMs of a sublayer run as one grouped launch, with
# ragged tiles in the ffn direction.
LM_MLP_MID = Workload("lm_mlp_mid", 300, 256, (Layer(SWIGLU, 256, 576), Layer(SWIGLU, 256, 576)),
                      1000, False, "bf16", "zipf", head_init="normal002", ignore_frac=0.05)

# More than 1024 rows with small widths: with the update registered, a step
# of this size applies it in the weight-gradient GEMMs' epilogues (smaller
# batches write u and update every tensor in one launch afterwards).
LM_MLP_K1100 = Workload("lm_mlp_k1100", 1100, 128, (Layer(SWIGLU, 128, 320), Layer(SWIGLU, 128, 320)),
                        777, False, "bf16", "zipf", head_init="normal002", ignore_frac=0.05)

# RMSNorm variants: an LM block whose head input is normalised (one SwiGLU
# sublayer, then the final norm, as in the paper's Qwen3 models), and an fp32
# MLP with a norm between two linear layers.
LM_NORM_SMALL = Workload("lm_norm_small", 260, 128, (Layer(SWIGLU, 128, 320), Layer(RMSNORM, 128, 128)),
                         777, False, "bf16", "zipf", head_init="normal002", ignore_frac=0.05)
TINY_NORM_F32 = Workload("tiny_norm_f32", 37, 29, (Layer(LINEAR_GELU, 29, 45, True), Layer(RMSNORM, 45, 45),
                                                    Layer(LINEAR, 45, 33, True)),
                         7, True, "f32", "uniform", steps=3, ignore_frac=0.1)
LM_NORM_BF16 = Workload("lm_norm_bf16", 16384, 2048,
                        (Layer(SWIGLU, 2048, 8192), Layer(SWIGLU, 2048, 8192), Layer(RMSNORM, 2048, 2048)),
                        32000, False, "bf16", "zipf", head_init="normal002")

WORKLOADS = {w.name: w for w in (TINY_MLP_F32, VISION_HEAD_BF16, LM_HEAD_BF16, LM_MLP_BF16,
                                  LM_HEAD_SMALL, LM_MLP_SMALL, VISION_SMALL, TINY_RAGGED_F32, LM_HEAD_WIDE,
                                  LM_NORM_SMALL, TINY_NORM_F32, LM_NORM_BF16, LM_MLP_MID, LM_MLP_K1100,
                                  VISION_MID, TINY_BF16, VISION_WIDE)}


# --------------------------------------------------------------------------
# Update sweep buffers
# --------------------------------------------------------------------------
def update_sweep_host(n: int, seed: int = 0):
    """theta, g (bf16 bits), h, v for the flat update sweep: N(0, 1e-3) values,
    v = (N(0, 1e-3))^2 >= 0."""
    g = _rng(seed, 3000)
    theta = g.standard_normal(n, dtype=np.float32) * np.float32(1e-3)
    grad = bf16_bits(g.standard_normal(n, dtype=np.float32) * np.float32(1e-3))
    h = g.standard_normal(n, dtype=np.float32) * np.float32(1e-3)
    z = g.standard_normal(n, dtype=np.float32) * np.float32(1e-3)
    v = z * z
    return theta, grad, h, v


def update_sweep_device(n: int, seed: int, device):
    """Same distribution as :func:`update_sweep_host`, drawn on the device with a
    seeded ``torch.Generator`` (used where the host would take too long)."""
    import torch
    gen = torch.Generator(device=device)
    gen.manual_seed(int(seed) * 7919 + 3000)
    theta = torch.randn(n, generator=gen, device=device, dtype=torch.float32).mul_(1e-3)
    grad = torch.randn(n, generator=gen, device=device, dtype=torch.float32).mul_(1e-3).to(torch.bfloat16)
    h = torch.randn(n, generator=gen, device=device, dtype=torch.float32).mul_(1e-3)
    v = torch.randn(n, generator=gen, device=device, dtype=torch.float32).mul_(1e-3).square_()
    return theta, grad, h, v
