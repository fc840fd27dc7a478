"""Seeded synthetic inputs shaped like the paper's workloads.

This module holds no part of the fake-quantizer's arithmetic: it only draws
random tensors (weights, activations, coefficients, upstream gradients) with
the shapes and value distributions of the layers FOCUS quantizes
(Sec. 4.1: Qwen3 and LLaMA-3 families, W4A4, calibration batches of
2,048-token sequences).  Both the CUDA path's tests and the oracle's tests
draw from here, so both sides always see the same bytes.

bfloat16 tensors are produced by drawing float32 values and keeping the high
16 bits of each (truncation): a valid way to obtain bf16 samples that does not
reuse any rounding routine of the method.  They are returned as uint16 bit
patterns on the host, or as torch.bfloat16 on a device.

Recipes (per tensor, seed = base seed + 16 * tensor index):
  weights      Student-t(nu) * scale, plus a few input columns (x30) or
               entries (x20) scaled up as outliers;
  activations  N(0, 1) with a few fixed hidden channels scaled up (x50);
  coefficients 1 + U(-j, j) or U(lo, hi) fp32;
  gradients    N(0, 1) in the tensor's dtype.
"""
from __future__ import annotations

import dataclasses
import math
from typing import List, Optional, Tuple

import numpy as np

# ----------------------------------------------------------------------------
# layer shapes ([out, in] weights; blocks run along `in`, the contiguous dim)
# ----------------------------------------------------------------------------
QWEN3_4B_LAYER = [  # hidden 2560, 32 q heads x 128, 8 kv heads x 128, MLP 9728
    ("q_proj", 4096, 2560), ("k_proj", 1024, 2560), ("v_proj", 1024, 2560),
    ("o_proj", 2560, 4096), ("gate_proj", 9728, 2560), ("up_proj", 9728, 2560),
    ("down_proj", 2560, 9728),
]
LLAMA3_8B_BLOCK = [  # hidden 4096, 32 q heads, 8 kv heads x 128, MLP 14336
    ("q_proj", 4096, 4096), ("k_proj", 1024, 4096), ("v_proj", 1024, 4096),
    ("o_proj", 4096, 4096), ("gate_proj", 14336, 4096), ("up_proj", 14336, 4096),
    ("down_proj", 4096, 14336),
]
LLAMA_70B_LAYER = [  # hidden 8192, 64 q heads, 8 kv heads x 128, MLP 28672
    ("q_proj", 8192, 8192), ("k_proj", 1024, 8192), ("v_proj", 1024, 8192),
    ("o_proj", 8192, 8192), ("gate_proj", 28672, 8192), ("up_proj", 28672, 8192),
    ("down_proj", 8192, 28672),
]


@dataclasses.dataclass(frozen=True)
class TensorSpec:
    name: str
    rows: int
    cols: int


@dataclasses.dataclass(frozen=True)
class Workload:
    """One configuration: a list of tensors plus how to draw them."""
    name: str
    tensors: Tuple[TensorSpec, ...]
    dtype: str                  # "f32", "bf16" or "f16"
    fmts: Tuple[str, ...]       # subset of ("mxfp4", "nvfp4")
    kind: str                   # "weight" or "activation"
    nu: Optional[float]         # Student-t degrees of freedom (weights)
    scale: float                # multiplier of the base draw
    outlier: str                # "entries", "in_cols", "channels", "none"
    outlier_count: float        # fraction (entries) or count (cols/channels)
    outlier_mult: float
    coef: Tuple[float, float]   # U(lo, hi) for crs and dgs
    seed: int

    @property
    def elements(self) -> int:
        return sum(t.rows * t.cols for t in self.tensors)


def _specs(lst):
    return tuple(TensorSpec(*t) for t in lst)


WORKLOADS = {
    # single 256x512 fp32 weight, MXFP4, per-block CRS + DGS(8)
    "w256x512_f32": Workload("w256x512_f32", _specs([("w", 256, 512)]), "f32", ("mxfp4",),
                             "weight", None, 0.02, "entries", 0.01, 20.0, (0.9, 1.1), 1000),
    # Qwen3-4B decoder layer, 7 projections, bf16, NVFP4
    "qwen3_4b_layer": Workload("qwen3_4b_layer", _specs(QWEN3_4B_LAYER), "bf16", ("nvfp4",),
                               "weight", 4.0, 0.02, "in_cols", 8, 30.0, (0.9, 1.1), 1001),
    # W4A4 activations: 128 sequences x 2048 tokens x hidden 4096
    "act_262144x4096": Workload("act_262144x4096", _specs([("act", 262144, 4096)]), "bf16",
                                ("mxfp4", "nvfp4"), "activation", None, 1.0, "channels", 6,
                                50.0, (0.9, 1.1), 1002),
    # LLaMA-3-8B decoder block, both formats, coefficients U(0.8, 1.2)
    "llama3_8b_block": Workload("llama3_8b_block", _specs(LLAMA3_8B_BLOCK), "bf16",
                                ("mxfp4", "nvfp4"), "weight", 5.0, 0.02 * math.sqrt(3.0 / 5.0),
                                "none", 0, 1.0, (0.8, 1.2), 1003),
    # 70B-shaped layer set, both formats
    "llama_70b_layer": Workload("llama_70b_layer", _specs(LLAMA_70B_LAYER), "bf16",
                                ("mxfp4", "nvfp4"), "weight", 5.0, 0.02 * math.sqrt(3.0 / 5.0),
                                "none", 0, 1.0, (0.9, 1.1), 1004),
}


def sweep_workload(nbytes: int) -> Workload:
    """A [n/8192, 8192] bf16 Gaussian tensor of `nbytes` bytes, 0.1% outliers x40."""
    n = nbytes // 2
    rows = max(1, n // 8192)
    return Workload(f"sweep_{nbytes}", (TensorSpec("x", rows, 8192),), "bf16",
                    ("mxfp4", "nvfp4"), "activation", None, 1.0, "entries", 0.001, 40.0,
                    (0.9, 1.1), 1005)


SWEEP_BYTES = [1 << k for k in range(20, 33)]  # 1 MB ... 4 GB (13 points)


# ----------------------------------------------------------------------------
# host (numpy) draws
# ----------------------------------------------------------------------------
def tensor_seed(w: Workload, idx: int, salt: int = 0) -> int:
    return w.seed + 16 * idx + salt


def to_bf16_bits(f32: np.ndarray) -> np.ndarray:
    """Keep the high half of each float32 (truncation) as uint16 bf16 bits."""
    f32 = np.ascontiguousarray(f32, dtype=np.float32)
    return (f32.view(np.uint32) >> 16).astype(np.uint16)


def bf16_bits_to_f32(b: np.ndarray) -> np.ndarray:
    return (b.astype(np.uint32) << 16).view(np.float32)


def draw_values(w: Workload, rows: int, cols: int, seed: int) -> np.ndarray:
    """float32 [rows, cols] input values following the workload's recipe."""
    rng = np.random.Generator(np.random.PCG64(seed))
    if w.nu is not None:
        v = rng.standard_t(w.nu, size=(rows, cols)) * w.scale
    else:
        v = rng.standard_normal(size=(rows, cols)) * w.scale
    if w.outlier == "entries" and w.outlier_count > 0 and rows * cols > 0:
        k = max(1, int(round(w.outlier_count * rows * cols)))
        idx = rng.choice(rows * cols, size=k, replace=False)
        v.reshape(-1)[idx] *= w.outlier_mult
    elif w.outlier in ("in_cols", "channels") and w.outlier_count > 0:
        k = min(cols, int(w.outlier_count))
        idx = rng.choice(cols, size=k, replace=False)
        v[:, idx] *= w.outlier_mult
    return v.astype(np.float32)


def draw_coefs(w: Workload, n: int, seed: int) -> np.ndarray:
    rng = np.random.Generator(np.random.PCG64(seed))
    lo, hi = w.coef
    return rng.uniform(lo, hi, size=n).astype(np.float32)


def draw_grad(rows: int, cols: int, seed: int) -> np.ndarray:
    rng = np.random.Generator(np.random.PCG64(seed))
    return rng.standard_normal(size=(rows, cols)).astype(np.float32)


def host_tensor(w: Workload, idx: int, rows: Optional[int] = None):
    """(x, g) host arrays for tensor `idx` (optionally only the first `rows`
    rows), in the workload's dtype: float32, uint16 bf16 bits, or float16
    (numpy's round-to-nearest conversion of the float32 draws)."""
    t = w.tensors[idx]
    r = t.rows if rows is None else min(rows, t.rows)
    x = draw_values(w, r, t.cols, tensor_seed(w, idx))
    g = draw_grad(r, t.cols, tensor_seed(w, idx, 1))
    if w.dtype == "bf16":
        return to_bf16_bits(x), to_bf16_bits(g)
    if w.dtype == "f16":
        return x.astype(np.float16), g.astype(np.float16)
    return x, g


def host_coefs(w: Workload, idx: int, block: int, sub: int, shared: bool = False,
               rows: Optional[int] = None):
    """(crs, dgs) fp32 arrays: [rows or 1, cols/block] and [rows or 1, cols/sub]."""
    t = w.tensors[idx]
    r = 1 if shared else (t.rows if rows is None else min(rows, t.rows))
    crs = draw_coefs(w, r * (t.cols // block), tensor_seed(w, idx, 2)).reshape(r, -1)
    dgs = draw_coefs(w, r * (t.cols // sub), tensor_seed(w, idx, 3)).reshape(r, -1)
    return crs, dgs


# ----------------------------------------------------------------------------
# device (torch) draws for sizes the host would take long to generate
# ----------------------------------------------------------------------------
def device_tensor(w: Workload, idx: int, device, torch_mod=None):
    """(x, g) torch tensors drawn directly on `device` with a seeded
    torch.Generator (Philox on CUDA).  Same recipe as host_tensor, different
    random stream; bf16 by truncation of float32 draws."""
    import torch
    t = w.tensors[idx]
    gen = torch.Generator(device=device)
    gen.manual_seed(tensor_seed(w, idx))
    shape = (t.rows, t.cols)
    if w.nu is not None and float(w.nu).is_integer():
        # Student-t(nu) = Z / sqrt(chi2_nu / nu), chi2_nu = sum of nu squared normals
        z = torch.randn(shape, generator=gen, device=device)
        chi = torch.zeros(shape, device=device)
        for _ in range(int(w.nu)):
            e = torch.randn(shape, generator=gen, device=device)
            chi.addcmul_(e, e)
        v = z / torch.sqrt(chi / w.nu)
        del chi
        v.mul_(w.scale)
    else:
        v = torch.randn(shape, generator=gen, device=device).mul_(w.scale)
    if w.outlier == "entries" and w.outlier_count > 0 and t.rows * t.cols > 0:
        k = max(1, int(round(w.outlier_count * t.rows * t.cols)))
        idx_ = torch.randint(0, t.rows * t.cols, (k,), generator=gen, device=device)
        v.view(-1)[idx_] *= w.outlier_mult
    elif w.outlier in ("in_cols", "channels") and w.outlier_count > 0:
        k = min(t.cols, int(w.outlier_count))
        cols = torch.randperm(t.cols, generator=gen, device=device)[:k]
        v[:, cols] *= w.outlier_mult
    gg = torch.Generator(device=device)
    gg.manual_seed(tensor_seed(w, idx, 1))
    g = torch.randn(shape, generator=gg, device=device)
    if w.dtype == "bf16":
        def trunc(a):
            return (a.view(torch.int32) >> 16).to(torch.int16).view(torch.bfloat16)
        return trunc(v), trunc(g)
    if w.dtype == "f16":
        return v.half(), g.half()
    return v, g


def device_coefs(w: Workload, idx: int, block: int, sub: int, device, shared: bool = False):
    import torch
    t = w.tensors[idx]
    r = 1 if shared else t.rows
    lo, hi = w.coef
    out = []
    for salt, n in ((2, t.cols // block), (3, t.cols // sub)):
        gen = torch.Generator(device=device)
        gen.manual_seed(tensor_seed(w, idx, salt))
        out.append(torch.rand((r, n), generator=gen, device=device) * (hi - lo) + lo)
    return out[0], out[1]
