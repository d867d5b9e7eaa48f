"""Seeded synthetic inputs for HLA workloads.

This module holds no arithmetic of the method: it only draws random tensors
with the distributions of the workloads and rounds them to the compute dtype.
Both the fp64 oracle and the CUDA path consume what it returns, so that parity
checks compare the two implementations on bit-identical inputs.

Recipe (every workload):
* q and k rows are drawn i.i.d. N(0, I_d) in float64 and then scaled to unit
  L2 norm; v entries are i.i.d. N(0, 1) in float64;
* the float64 values are rounded to the workload dtype (bf16: round to
  nearest-even through float32; f32: plain float32 rounding);
* generation uses numpy's PCG64 generator seeded with the workload seed, in
  the order q, k, v, tensor by tensor, head-major ([B, H, n, d] contiguous).

Arrays are returned as float32 numpy arrays whose values are exactly
representable in the workload dtype; ``as_torch`` turns them into tensors of
that dtype without further rounding.
"""
from __future__ import annotations

from dataclasses import dataclass

import numpy as np


@dataclass(frozen=True)
class Workload:
    name: str
    B: int
    H: int
    n: int
    d: int
    dv: int
    chunk: int
    dtype: str          # "f32" or "bf16"
    masked: bool
    normalized: bool
    seed: int
    order: int = 2      # 2 = second-order HLA, 3 = third-order HLA, 22 = asymmetric second order (AHLA)
    decode_prefix: int = 0
    decode_steps: int = 0

    @property
    def BH(self) -> int:
        return self.B * self.H


# The five workloads of the build: shapes, dtypes and flags of the paper's
# operator as it is exercised here.  Seeds are fixed per workload.
WORKLOADS = {
    "tiny_f32": Workload("tiny_f32", 1, 1, 64, 16, 16, 16, "f32", True, False, 0),
    "mid_bf16": Workload("mid_bf16", 8, 16, 2048, 64, 64, 64, "bf16", True, False, 1),
    "long_bf16_norm": Workload("long_bf16_norm", 2, 16, 16384, 128, 128, 128, "bf16", True, True, 2),
    "decode_bf16": Workload("decode_bf16", 64, 32, 0, 128, 128, 128, "bf16", True, False, 3,
                            decode_prefix=4096, decode_steps=256),
    "hla3_f32": Workload("hla3_f32", 4, 8, 4096, 32, 32, 32, "f32", True, False, 4, order=3),
    # asymmetric second order (AHLA) at the shapes of the d = 64 forward, and its decode step at the
    # shapes of the second-order decode workload
    "ahla_bf16": Workload("ahla_bf16", 8, 16, 2048, 64, 64, 64, "bf16", True, False, 5, order=22),
    "ahla_decode_bf16": Workload("ahla_decode_bf16", 64, 32, 0, 128, 128, 64, "bf16", True, False, 6, order=22,
                                 decode_prefix=4096, decode_steps=256),
}

EPS = 1e-6  # the stability constant of the ratio-normalised output, used on both sides


def round_to(x: np.ndarray, dtype: str) -> np.ndarray:
    """Round float64 values to ``dtype`` and return them as float32."""
    x32 = np.asarray(x, dtype=np.float32)
    if dtype == "f32":
        return x32
    if dtype != "bf16":
        raise ValueError(dtype)
    bits = x32.view(np.uint32).astype(np.uint64)
    # round to nearest, ties to even, on the upper 16 bits (finite inputs only)
    bias = np.uint64(0x7FFF) + ((bits >> np.uint64(16)) & np.uint64(1))
    rounded = ((bits + bias) >> np.uint64(16)) << np.uint64(16)
    return rounded.astype(np.uint32).view(np.float32)


def _unit_rows(rng, shape):
    x = rng.standard_normal(shape)
    return x / np.linalg.norm(x, axis=-1, keepdims=True)


def make_qkv(B: int, H: int, n: int, d: int, dv: int, seed: int, dtype: str = "bf16"):
    """q, k: unit-norm Gaussian rows; v: N(0,1); shapes [B, H, n, d|dv]."""
    rng = np.random.default_rng(seed)
    q = round_to(_unit_rows(rng, (B, H, n, d)), dtype)
    k = round_to(_unit_rows(rng, (B, H, n, d)), dtype)
    v = round_to(rng.standard_normal((B, H, n, dv)), dtype)
    return q, k, v


def make_workload(w: Workload, n: int | None = None):
    """Inputs of a forward workload (optionally with a different n)."""
    return make_qkv(w.B, w.H, w.n if n is None else n, w.d, w.dv, w.seed, w.dtype)


def make_decode(w: Workload, prefix: int | None = None, steps: int | None = None):
    """Prefix tokens [B,H,prefix,*] and decode tokens [steps,B,H,*] of a decode workload.

    The prefix is drawn first and the decode tokens after it, from one stream.
    """
    prefix = w.decode_prefix if prefix is None else prefix
    steps = w.decode_steps if steps is None else steps
    rng = np.random.default_rng(w.seed)
    qp = round_to(_unit_rows(rng, (w.B, w.H, prefix, w.d)), w.dtype)
    kp = round_to(_unit_rows(rng, (w.B, w.H, prefix, w.d)), w.dtype)
    vp = round_to(rng.standard_normal((w.B, w.H, prefix, w.dv)), w.dtype)
    qs = round_to(_unit_rows(rng, (steps, w.B, w.H, w.d)), w.dtype)
    ks = round_to(_unit_rows(rng, (steps, w.B, w.H, w.d)), w.dtype)
    vs = round_to(rng.standard_normal((steps, w.B, w.H, w.dv)), w.dtype)
    return (qp, kp, vp), (qs, ks, vs)


def as_torch(x: np.ndarray, dtype: str, device=None):
    """float32 array of ``dtype``-exact values -> torch tensor of that dtype."""
    import torch
    t = torch.from_numpy(np.ascontiguousarray(x))
    t = t.to(torch.bfloat16) if dtype == "bf16" else t.to(torch.float32)
    return t.to(device) if device is not None else t
