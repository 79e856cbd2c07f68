"""Seeded synthetic workloads for the PBB decode step and the whole-sequence forward.

This module only draws numbers: it holds none of the method's arithmetic (no
support, no slot mapping, no attention). Both the CUDA path's tests and the
oracle take their inputs from here, so the two see the same bytes.

Every value is N(0, 1) from a seeded ``torch.Generator`` and then cast to the
workload's dtype. A workload starts each sequence at a position ``t0``; the
history window holds the B tokens before it (positions t0-B .. t0-1, zero rows
for positions below 0, which do not exist), and every decode step brings one new
query/key/value per sequence. The outlier workload multiplies each K and V
element by 20 with probability 1 %.

The recipes mirror the paper's efficiency protocol (seeded synthetic inputs,
no dataset; Sec. 5 and Appendix F.2) at the shapes of the five benchmark
configurations of this package.
"""
from __future__ import annotations

from dataclasses import dataclass, replace
from typing import Optional, Tuple

import torch

__all__ = ["Workload", "WORKLOADS", "sweep_workload", "start_positions", "history_window",
           "step_inputs", "torch_dtype", "SequenceWorkload", "FORWARD_WORKLOADS", "sequence_inputs"]


@dataclass(frozen=True)
class Workload:
    name: str
    batch: int
    Hq: int
    Hkv: int
    d: int
    B: int
    dtype: str                 # "bf16" or "f32"
    steps: int
    t0_lo: int = 0             # t0 ~ U[t0_lo, t0_hi) per sequence; t0_hi == t0_lo + 1 -> aligned
    t0_hi: int = 1
    outlier_frac: float = 0.0
    outlier_scale: float = 1.0
    seed: int = 0

    @property
    def group(self) -> int:
        return self.Hq // self.Hkv

    @property
    def elem_bytes(self) -> int:
        return 2 if self.dtype == "bf16" else 4

    def with_(self, **kw) -> "Workload":
        return replace(self, **kw)


WORKLOADS = {
    # fp32, one layer, 1024 sequential steps from t = 0 (8 block boundaries)
    "fp32_b1_B128": Workload("fp32_b1_B128", batch=1, Hq=8, Hkv=2, d=64, B=128, dtype="f32",
                             steps=1024, t0_lo=0, t0_hi=1, seed=0),
    # bf16, aligned sequences, 4096 steps sweeping every phase of 4 blocks
    "bf16_b32_B1024": Workload("bf16_b32_B1024", batch=32, Hq=16, Hkv=4, d=128, B=1024,
                               dtype="bf16", steps=4096, t0_lo=0, t0_hi=1, seed=1),
    # bf16, ragged positions t0 ~ U[0, 512K), ring pre-filled
    "bf16_b64_B2048_ragged": Workload("bf16_b64_B2048_ragged", batch=64, Hq=32, Hkv=8, d=128,
                                      B=2048, dtype="bf16", steps=256, t0_lo=0,
                                      t0_hi=512 * 1024, seed=2),
    # bf16, GQA group 8, 1 % of K/V entries scaled x20, t0 ~ U[0, 64K)
    "bf16_b256_B4096_outlier": Workload("bf16_b256_B4096_outlier", batch=256, Hq=16, Hkv=2,
                                        d=128, B=4096, dtype="bf16", steps=128, t0_lo=0,
                                        t0_hi=64 * 1024, outlier_frac=0.01, outlier_scale=20.0,
                                        seed=3),
}

SWEEP_BATCHES = (1, 8, 64, 512)
SWEEP_BLOCKS = (512, 1024, 2048, 4096)


def sweep_workload(batch: int, B: int, steps: int = 256) -> Workload:
    """Steady-state throughput point: Hq 32, Hkv 8, d 128, bf16, t0 ~ U[B, 2^20)."""
    return Workload(f"sweep_b{batch}_B{B}", batch=batch, Hq=32, Hkv=8, d=128, B=B, dtype="bf16",
                    steps=steps, t0_lo=B, t0_hi=1 << 20, seed=4 + batch * 7919 + B)


def torch_dtype(w: Workload) -> torch.dtype:
    return torch.bfloat16 if w.dtype == "bf16" else torch.float32


def _gen(device, seed: int, *tags: int) -> torch.Generator:
    h = seed & 0xFFFFFFFF
    for x in tags:  # a fixed mixing of the tags into one 63-bit seed
        h = (h * 0x9E3779B97F4A7C15 + (x & 0xFFFFFFFFFFFF) + 0x632BE59BD9B4E019) & ((1 << 63) - 1)
    g = torch.Generator(device=device)
    g.manual_seed(h)
    return g


def _normal(shape, w: Workload, device, *tags: int, outliers: bool = False) -> torch.Tensor:
    x = torch.randn(shape, generator=_gen(device, w.seed, *tags), device=device,
                    dtype=torch.float32)
    if outliers and w.outlier_frac > 0:
        u = torch.rand(shape, generator=_gen(device, w.seed, *tags, 7), device=device)
        x = torch.where(u < w.outlier_frac, x * w.outlier_scale, x)
    return x.to(torch_dtype(w))


def start_positions(w: Workload, device="cpu") -> torch.Tensor:
    """Per-sequence start position t0 (int64 [batch])."""
    if w.t0_hi <= w.t0_lo + 1:
        return torch.full((w.batch,), w.t0_lo, dtype=torch.int64, device=device)
    return torch.randint(w.t0_lo, w.t0_hi, (w.batch,), generator=_gen("cpu", w.seed, 1),
                         dtype=torch.int64).to(device)


def history_window(w: Workload, t0: torch.Tensor, device="cpu",
                   rows: Optional[int] = None) -> Tuple[torch.Tensor, torch.Tensor]:
    """K/V of the `rows` (default B) positions before t0: [batch, Hkv, rows, d].

    Row j holds position t0 - rows + j; rows at negative positions are zero.
    """
    n = w.B if rows is None else rows
    shape = (w.batch, w.Hkv, n, w.d)
    k = _normal(shape, w, device, 2, outliers=True)
    v = _normal(shape, w, device, 3, outliers=True)
    pos = t0.to(device).view(-1, 1) - n + torch.arange(n, device=device).view(1, -1)
    keep = (pos >= 0).view(w.batch, 1, n, 1)
    zero = torch.zeros((), dtype=k.dtype, device=device)
    return torch.where(keep, k, zero), torch.where(keep, v, zero)


def step_inputs(w: Workload, step: int, device="cpu") -> Tuple[torch.Tensor, torch.Tensor, torch.Tensor]:
    """(q [batch, Hq, d], k_new [batch, Hkv, d], v_new [batch, Hkv, d]) of decode step `step`."""
    q = _normal((w.batch, w.Hq, w.d), w, device, 10, step)
    k = _normal((w.batch, w.Hkv, w.d), w, device, 11, step, outliers=True)
    v = _normal((w.batch, w.Hkv, w.d), w, device, 12, step, outliers=True)
    return q, k, v


def step_inputs_stacked(w: Workload, steps: int, device="cpu", first: int = 0):
    """Stacked inputs of `steps` consecutive decode steps: ([steps, ...] x 3)."""
    qs, ks, vs = zip(*(step_inputs(w, first + i, device) for i in range(steps)))
    return torch.stack(qs), torch.stack(ks), torch.stack(vs)


@dataclass(frozen=True)
class SequenceWorkload:
    """Whole sequences for the forward pass: q [batch, Hq, n, d], k/v [batch, Hkv, n, d], bf16."""
    name: str
    batch: int
    Hq: int
    Hkv: int
    d: int
    B: int
    n: int
    outlier_frac: float = 0.0
    outlier_scale: float = 1.0
    seed: int = 0
    dtype: str = "bf16"

    @property
    def group(self) -> int:
        return self.Hq // self.Hkv

    def with_(self, **kw) -> "SequenceWorkload":
        return replace(self, **kw)


FORWARD_WORKLOADS = {
    # the paper's local-layer geometry (head dim 64, block 128) at 8K context, group 4
    "fwd_b16_n8192_B128": SequenceWorkload("fwd_b16_n8192_B128", batch=16, Hq=8, Hkv=2, d=64, B=128,
                                           n=8192, seed=40),
    # the decode benchmark's heads (Hq 32, Hkv 8, d 128) with 4096-token blocks at 32K context
    "fwd_b2_n32768_B4096": SequenceWorkload("fwd_b2_n32768_B4096", batch=2, Hq=32, Hkv=8, d=128, B=4096,
                                            n=32768, seed=41),
}


def sequence_inputs(w: SequenceWorkload, device="cpu") -> Tuple[torch.Tensor, torch.Tensor, torch.Tensor]:
    """(q [batch, Hq, n, d], k [batch, Hkv, n, d], v [batch, Hkv, n, d]) of a sequence workload."""
    q = _normal((w.batch, w.Hq, w.n, w.d), w, device, 20)
    k = _normal((w.batch, w.Hkv, w.n, w.d), w, device, 21, outliers=True)
    v = _normal((w.batch, w.Hkv, w.n, w.d), w, device, 22, outliers=True)
    return q, k, v
