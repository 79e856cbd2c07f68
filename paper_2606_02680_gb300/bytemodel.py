"""Algorithmic bytes and FLOPs of one PBB (or sliding-window) decode step, for
roofline reporting.

Support size (Sec. 3, Eq. pbb; Appendix F.1, Eq. pbb_cache_support): with
B = 2h, p = B*floor(t/B), r = t - p,
    |A(t)| = (r + 1) + h   if p > 0 and r < h,   else r + 1.

Bytes one step must move for a sequence (the current token is read from
k_new/v_new, not from the ring):
    Hkv * d * e * [2 (|A| - 1)      K and V of the ring slots read
                   + 2              k_new, v_new read
                   + 2]             ring slot r written (K and V)
  + Hq * d * e                      q read
  + Hq * d * 4                      fp32 output written
  + 4                               pos read
with e the element size. FLOPs: 4 d |A| per query head (2 for q.k, 2 for p.v;
Appendix A.5 counts about 4 d_h E).
"""
from __future__ import annotations

import numpy as np


def support_size(t, B: int, window: int | None = None):
    """|A(t)| of PBB with block B, or of the sliding window {t-w+1, ..., t} (min(t+1, w))."""
    t = np.asarray(t, dtype=np.int64)
    if window is not None:
        return np.minimum(t + 1, window)
    h = B // 2
    p = (t // B) * B
    r = t - p
    return r + 1 + np.where((p > 0) & (r < h), h, 0)


def step_bytes(t, Hq: int, Hkv: int, d: int, B: int, elem_bytes: int, window: int | None = None) -> int:
    """Algorithmic bytes of one decode step over sequences at positions t."""
    a = support_size(t, B, window)
    per_seq = Hkv * d * elem_bytes * (2 * (a - 1) + 4) + Hq * d * elem_bytes + Hq * d * 4 + 4
    return int(per_seq.sum())


def step_flops(t, Hq: int, d: int, B: int, window: int | None = None) -> int:
    return int((4 * d * Hq * support_size(t, B, window)).sum())


def mean_support(B: int) -> float:
    """Phase-average support at steady state, (3h + 1)/2."""
    h = B // 2
    return (3 * h + 1) / 2
