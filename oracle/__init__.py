"""fp64 CPU oracle for Post-Boundary Bridge (PBB) attention: the decode step and
the whole-sequence forward.

TEST INFRASTRUCTURE ONLY: the tests, ``__graft_entry__.smoke()`` and the
benchmark's CPU-baseline leg may import this package; the product path
(``paper_2606_02680_gb300``) never does. The oracle shares no code with the
CUDA library and neither imports the other.

The arithmetic lives in ``pbb_oracle.c`` (plain C, fp64, OpenMP over
sequences); this module compiles it with gcc on first use and marshals numpy
arrays. What each function computes is stated in the C file and below:

* ``in_support``       Eq. (pbb), Sec. 3, block/bridge form.
* ``support_count``    |A_PBB(t)| by testing every s in [0, t].
* ``attend``           Eq. (attention), brute force over a history window.
* ``RingSim``          the relocation-free ring of Appendix F.1 (slot s mod b)
                       and a ring-indexed second evaluation over [a(t), t].
* ``in_window``, ``window_count``, ``attend_window``
                       sliding-window attention (Sec. 2.3), the comparison pattern.
* ``forward``          PBB attention for every position of whole sequences (the
                       forward pass / prefill), with the log-partition of Eq. (lse).
* ``backward``         its gradients with respect to q, k and v.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "pbb_oracle.c")
_BUILD = os.path.join(_HERE, "_build")
_LIB_PATH = os.path.join(_BUILD, "liboracle.so")
_lock = threading.Lock()
_lib = None

ORACLE_OK = 0
ORACLE_ERR_ARG = -1
ORACLE_ERR_WINDOW = -2
ORACLE_ERR_RING = -3


class OracleError(RuntimeError):
    pass


def build(force: bool = False) -> str:
    """Compile the oracle into ``oracle/_build/liboracle.so`` (gcc, -O2, OpenMP)."""
    os.makedirs(_BUILD, exist_ok=True)
    if force or not os.path.exists(_LIB_PATH) or os.path.getmtime(_LIB_PATH) < os.path.getmtime(_SRC):
        tmp = _LIB_PATH + f".tmp{os.getpid()}"
        cmd = ["gcc", "-O2", "-fopenmp", "-fPIC", "-shared", "-std=c11", "-Wall", "-Wextra",
               "-o", tmp, _SRC, "-lm"]
        subprocess.run(cmd, check=True)
        os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


def _load():
    global _lib
    with _lock:
        if _lib is not None:
            return _lib
        lib = ctypes.CDLL(build())
        L, I, P = ctypes.c_long, ctypes.c_int, ctypes.c_void_p
        lib.pbb_oracle_in_support.argtypes = [L, L, L]
        lib.pbb_oracle_in_support.restype = I
        lib.pbb_oracle_support_count.argtypes = [L, L]
        lib.pbb_oracle_support_count.restype = L
        lib.pbb_oracle_attend.argtypes = [P, P, P, P, P, L, I, I, I, I, L, P, I]
        lib.pbb_oracle_attend.restype = I
        lib.pbb_oracle_ring_append.argtypes = [P, P, P, P, I, I, L, L]
        lib.pbb_oracle_ring_append.restype = None
        lib.pbb_oracle_ring_replay.argtypes = [P, P, P, P, L, I, I, L, L]
        lib.pbb_oracle_ring_replay.restype = None
        lib.pbb_oracle_attend_ring.argtypes = [P, P, P, P, I, P, I, I, I, I, L, P, I]
        lib.pbb_oracle_attend_ring.restype = I
        lib.pbb_oracle_in_window.argtypes = [L, L, L]
        lib.pbb_oracle_in_window.restype = I
        lib.pbb_oracle_window_count.argtypes = [L, L]
        lib.pbb_oracle_window_count.restype = L
        lib.pbb_oracle_attend_window.argtypes = [P, P, P, P, P, L, I, I, I, I, L, P, I]
        lib.pbb_oracle_attend_window.restype = I
        lib.pbb_oracle_forward_rows.argtypes = [P, P, P, I, I, I, L, I, L, P, L, P, P, I]
        lib.pbb_oracle_forward_rows.restype = I
        lib.pbb_oracle_backward.argtypes = [P, P, P, P, I, I, I, L, I, L, P, P, P, I]
        lib.pbb_oracle_backward.restype = I
        lib.pbb_oracle_max_threads.argtypes = []
        lib.pbb_oracle_max_threads.restype = I
        _lib = lib
        return lib


def _ptr(a: np.ndarray) -> ctypes.c_void_p:
    return ctypes.c_void_p(a.ctypes.data)


def _f64(a) -> np.ndarray:
    """Exact widening to a C-contiguous fp64 array (accepts numpy or torch CPU tensors)."""
    if hasattr(a, "detach"):
        a = a.detach().to("cpu").double().numpy()
    return np.ascontiguousarray(a, dtype=np.float64)


def _bits(a) -> np.ndarray:
    """Raw element bits of a bf16/fp32 tensor as a contiguous uint8 array."""
    if hasattr(a, "detach"):
        import torch

        t = a.detach().to("cpu").contiguous()
        if t.dtype == torch.bfloat16:
            return t.view(torch.int16).numpy().view(np.uint8).reshape(*t.shape[:-1], -1)
        if t.dtype == torch.float32:
            return t.view(torch.int32).numpy().view(np.uint8).reshape(*t.shape[:-1], -1)
        raise TypeError(f"unsupported dtype {t.dtype}")
    a = np.ascontiguousarray(a)
    if a.dtype == np.float32:
        return a.view(np.uint8).reshape(*a.shape[:-1], -1)
    if a.dtype == np.uint16:
        return a.view(np.uint8).reshape(*a.shape[:-1], -1)
    raise TypeError(f"unsupported dtype {a.dtype}")


def max_threads() -> int:
    return int(_load().pbb_oracle_max_threads())


def in_support(t: int, s: int, b: int) -> bool:
    """Eq. (pbb): whether source position s is in A_PBB(t) for block size b."""
    return bool(_load().pbb_oracle_in_support(t, s, b))


def support_count(t: int, b: int) -> int:
    """|A_PBB(t)| counted by brute force over s in [0, t]."""
    return int(_load().pbb_oracle_support_count(t, b))


def attend(q, hist_k, hist_v, s0, t, b: int, n_threads: int = 0) -> np.ndarray:
    """Brute-force PBB attention for one decode step (Eq. attention over Eq. pbb).

    q: [batch, Hq, d]; hist_k, hist_v: [batch, Hkv, n_hist, d] with row j holding
    position s0[b] + j; s0, t: [batch] integers. Returns fp64 [batch, Hq, d].
    """
    q = _f64(q)
    hk = _f64(hist_k)
    hv = _f64(hist_v)
    batch, Hq, d = q.shape
    _, Hkv, n_hist, d2 = hk.shape
    assert d2 == d and hv.shape == hk.shape and hk.shape[0] == batch
    s0a = np.ascontiguousarray(np.broadcast_to(np.asarray(s0, dtype=np.int64), (batch,)))
    ta = np.ascontiguousarray(np.broadcast_to(np.asarray(t, dtype=np.int64), (batch,)))
    out = np.zeros((batch, Hq, d), dtype=np.float64)
    rc = _load().pbb_oracle_attend(_ptr(q), _ptr(hk), _ptr(hv), _ptr(s0a), _ptr(ta), n_hist,
                                   batch, Hq, Hkv, d, b, _ptr(out), n_threads)
    if rc != ORACLE_OK:
        raise OracleError(f"pbb_oracle_attend returned {rc}")
    return out


def in_window(t: int, s: int, w: int) -> bool:
    """Sliding window (Sec. 2.3): s in {max(0, t-w+1), ..., t}."""
    return bool(_load().pbb_oracle_in_window(t, s, w))


def window_count(t: int, w: int) -> int:
    return int(_load().pbb_oracle_window_count(t, w))


def attend_window(q, hist_k, hist_v, s0, t, w: int, n_threads: int = 0) -> np.ndarray:
    """Brute-force sliding-window attention (window w, current position included);
    same arguments and layout as ``attend``."""
    q = _f64(q)
    hk = _f64(hist_k)
    hv = _f64(hist_v)
    batch, Hq, d = q.shape
    _, Hkv, n_hist, d2 = hk.shape
    assert d2 == d and hv.shape == hk.shape and hk.shape[0] == batch
    s0a = np.ascontiguousarray(np.broadcast_to(np.asarray(s0, dtype=np.int64), (batch,)))
    ta = np.ascontiguousarray(np.broadcast_to(np.asarray(t, dtype=np.int64), (batch,)))
    out = np.zeros((batch, Hq, d), dtype=np.float64)
    rc = _load().pbb_oracle_attend_window(_ptr(q), _ptr(hk), _ptr(hv), _ptr(s0a), _ptr(ta), n_hist,
                                          batch, Hq, Hkv, d, w, _ptr(out), n_threads)
    if rc != ORACLE_OK:
        raise OracleError(f"pbb_oracle_attend_window returned {rc}")
    return out


def forward(q, k, v, b: int, rows=None, n_threads: int = 0):
    """PBB attention for whole sequences (Sec. 3, Eq. attention over A_PBB(t) for every t).

    q: [batch, Hq, n, d]; k, v: [batch, Hkv, n, d] (row s = position s). rows: None for every
    (sequence, head, position), else an int array [n_rows, 3] of (sequence, query head, t).
    Returns (out, lse): out [batch, Hq, n, d] and lse [batch, Hq, n] for rows=None, else
    [n_rows, d] and [n_rows]; lse = ln sum_{s in A(t)} exp(z_ts) (natural log).
    """
    q = _f64(q)
    kk = _f64(k)
    vv = _f64(v)
    batch, Hq, n, d = q.shape
    _, Hkv, n2, d2 = kk.shape
    assert n2 == n and d2 == d and vv.shape == kk.shape and kk.shape[0] == batch
    full = rows is None
    if full:
        bi, j, t = np.meshgrid(np.arange(batch), np.arange(Hq), np.arange(n), indexing="ij")
        rows = np.stack([bi.ravel(), j.ravel(), t.ravel()], axis=1)
    rows = np.ascontiguousarray(np.asarray(rows, dtype=np.int64).reshape(-1, 3))
    out = np.zeros((rows.shape[0], d), dtype=np.float64)
    lse = np.zeros(rows.shape[0], dtype=np.float64)
    rc = _load().pbb_oracle_forward_rows(_ptr(q), _ptr(kk), _ptr(vv), batch, Hq, Hkv, n, d, b,
                                         _ptr(rows), rows.shape[0], _ptr(out), _ptr(lse), n_threads)
    if rc != ORACLE_OK:
        raise OracleError(f"pbb_oracle_forward_rows returned {rc}")
    if full:
        return out.reshape(batch, Hq, n, d), lse.reshape(batch, Hq, n)
    return out, lse


def backward(q, k, v, dout, b: int, n_threads: int = 0):
    """Gradients (dq, dk, dv) of the whole-sequence PBB attention for the upstream gradient
    dout [batch, Hq, n, d] (chain rule through Eq. attention over A_PBB(t)); fp64."""
    q = _f64(q)
    kk = _f64(k)
    vv = _f64(v)
    do = _f64(dout)
    batch, Hq, n, d = q.shape
    _, Hkv, n2, d2 = kk.shape
    assert n2 == n and d2 == d and vv.shape == kk.shape and do.shape == q.shape
    dq = np.zeros_like(q)
    dk = np.zeros_like(kk)
    dv = np.zeros_like(vv)
    rc = _load().pbb_oracle_backward(_ptr(q), _ptr(kk), _ptr(vv), _ptr(do), batch, Hq, Hkv, n, d, b,
                                     _ptr(dq), _ptr(dk), _ptr(dv), n_threads)
    if rc != ORACLE_OK:
        raise OracleError(f"pbb_oracle_backward returned {rc}")
    return dq, dk, dv


class RingSim:
    """Ring simulator of Appendix F.1: position s is stored in slot s mod b.

    Holds the raw element bits of K and V rings, shaped [batch, Hkv, b, row_bytes],
    and the position tag of every slot ([batch, b], -1 = never written). A
    fresh ring is all zero bytes, like a zero-initialised device ring.
    """

    def __init__(self, batch: int, Hkv: int, d: int, b: int, elem_bytes: int):
        assert elem_bytes in (2, 4)
        self.batch, self.Hkv, self.d, self.b, self.elem_bytes = batch, Hkv, d, b, elem_bytes
        self.row_bytes = d * elem_bytes
        self.k = np.zeros((batch, Hkv, b, self.row_bytes), dtype=np.uint8)
        self.v = np.zeros_like(self.k)
        self.tags = np.full((batch, b), -1, dtype=np.int64)

    def append(self, k_new, v_new, t) -> None:
        """Store the rows of position t[b] (k_new, v_new: [batch, Hkv, d]) at slot t mod b."""
        kb, vb = _bits(k_new), _bits(v_new)
        assert kb.shape == (self.batch, self.Hkv, self.row_bytes)
        ta = np.ascontiguousarray(np.broadcast_to(np.asarray(t, dtype=np.int64), (self.batch,)))
        lib = _load()
        for ring, rows in ((self.k, kb), (self.v, vb)):
            rows = np.ascontiguousarray(rows)
            lib.pbb_oracle_ring_append(_ptr(ring), _ptr(self.tags), _ptr(rows), _ptr(ta),
                                       self.batch, self.Hkv, self.b, self.row_bytes)

    def replay(self, hist_k, hist_v, s0) -> None:
        """Append a history window oldest first; row j of hist is position s0[b] + j."""
        kb, vb = _bits(hist_k), _bits(hist_v)
        n_hist = kb.shape[2]
        s0a = np.ascontiguousarray(np.broadcast_to(np.asarray(s0, dtype=np.int64), (self.batch,)))
        lib = _load()
        tags_k = self.tags.copy()
        for ring, rows in ((self.k, kb), (self.v, vb)):
            self.tags[:] = tags_k
            rows = np.ascontiguousarray(rows)
            lib.pbb_oracle_ring_replay(_ptr(ring), _ptr(self.tags), _ptr(rows), _ptr(s0a), n_hist,
                                       self.batch, self.Hkv, self.b, self.row_bytes)

    def attend(self, q, t, n_threads: int = 0) -> np.ndarray:
        """Attention over [a(t), t] read from the ring (which must already hold t)."""
        q = _f64(q)
        batch, Hq, d = q.shape
        assert batch == self.batch and d == self.d
        ta = np.ascontiguousarray(np.broadcast_to(np.asarray(t, dtype=np.int64), (batch,)))
        out = np.zeros((batch, Hq, d), dtype=np.float64)
        rc = _load().pbb_oracle_attend_ring(_ptr(q), _ptr(self.k), _ptr(self.v), _ptr(self.tags),
                                            self.elem_bytes, _ptr(ta), batch, Hq, self.Hkv, d,
                                            self.b, _ptr(out), n_threads)
        if rc != ORACLE_OK:
            raise OracleError(f"pbb_oracle_attend_ring returned {rc}")
        return out
