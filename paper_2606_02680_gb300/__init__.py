"""Python binding of libpbb, the GB300 decode step of Post-Boundary Bridge attention.

Argument marshalling only: every step of the computation runs in the CUDA
kernels of ``libpbb.so`` (built in-tree by ``build.py``), reached through the
C ABI of ``include/pbb.h`` with ctypes. PyTorch provides device memory and
streams. There is no CPU fallback: if the library is missing or no GPU is
visible, the calls raise.

Names follow the C ABI:

* ``ring_bytes``, ``ring_alloc`` / ``Rings``   the B-slot K/V rings (Appendix F.1)
* ``ring_prefill``                             load a ring from a history window
* ``decode_step``                              append + attention over A(t) (Sec. 3)
* ``decode_step_layers``                       one step of L layers in one launch
* ``swa_decode_step``                          the sliding-window control over the same rings
* ``forward``, ``ring_from_sequence``          whole-sequence PBB attention (prefill / training
                                               forward) and the rings it leaves for decoding
* ``backward``                                 its gradients dq, dk, dv
* ``decode_step_host``, ``HostPipeline``       the same with host-resident inputs/outputs
                                               (one at a time / overlapped across steps)
* ``advance_positions``, ``get_device_status``, ``reserve_workspace``,
  ``set_wait_timeout_ns``, ``set_chunk_keys``, ``plan_chunk_keys``
"""
from __future__ import annotations

import ctypes
import os
import threading

import torch

__all__ = [
    "PBB_OK", "PBB_ERR_INVALID_ARG", "PBB_ERR_UNSUPPORTED", "PBB_ERR_CUDA",
    "PBB_ERR_DEVICE_TIMEOUT", "PBB_ERR_WORKSPACE", "PBB_ERR_DEVICE_POSITION",
    "PBB_ERR_SCRATCH_LIMIT", "PbbError",
    "lib", "lib_path", "set_kernel", "plan_forward", "ring_bytes", "ring_alloc", "Rings", "ring_prefill", "decode_step", "decode_step_layers", "swa_decode_step", "forward", "backward", "ring_from_sequence",
    "decode_step_host", "HostPipeline", "advance_positions", "get_device_status", "reserve_workspace",
    "set_wait_timeout_ns", "set_chunk_keys", "plan_chunk_keys", "plan_kernel", "error_string", "stream_read",
    "EXPORTS",
]

PBB_OK = 0
PBB_ERR_INVALID_ARG = -1
PBB_ERR_UNSUPPORTED = -2
PBB_ERR_CUDA = -3
PBB_ERR_DEVICE_TIMEOUT = -4
PBB_ERR_WORKSPACE = -5
PBB_ERR_DEVICE_POSITION = -6
PBB_ERR_SCRATCH_LIMIT = -7

PBB_BF16 = 0
PBB_F32 = 1

# Every symbol include/pbb.h declares, with its ctypes signature.
_P, _I, _SZ, _ULL = ctypes.c_void_p, ctypes.c_int, ctypes.c_size_t, ctypes.c_ulonglong
EXPORTS = {
    "pbb_ring_bytes": (_SZ, [_I, _I, _I, _I, _I]),
    "pbb_ring_alloc": (_I, [ctypes.POINTER(_P), ctypes.POINTER(_P), _I, _I, _I, _I, _I, _P]),
    "pbb_ring_free": (_I, [_P, _P, _P]),
    "pbb_ring_prefill": (_I, [_P, _P, _P, _P, _P, _I, _I, _I, _I, _I, _P]),
    "pbb_reserve_workspace": (_I, [_I, _I, _I, _I, _I, _I, _P]),
    "pbb_decode_step": (_I, [_P, _P, _P, _P, _P, _P, _P, _I, _I, _I, _I, _I, _P]),
    "pbb_decode_step_f32": (_I, [_P, _P, _P, _P, _P, _P, _P, _I, _I, _I, _I, _I, _P]),
    "pbb_decode_step_noalloc": (_I, [_P, _P, _P, _P, _P, _P, _P, _I, _I, _I, _I, _I, _P]),
    "pbb_swa_decode_step": (_I, [_P, _P, _P, _P, _P, _P, _P, _I, _I, _I, _I, _I, _I, _I, _P]),
    "pbb_decode_step_layers": (_I, [_P, _P, _P, _P, _P, _P, _P, _I, _I, _I, _I, _I, _I, _I, _P]),
    "pbb_forward": (_I, [_P, _P, _P, _P, _P, _I, _I, _I, _I, _I, _I, _I, _P]),
    "pbb_plan_forward": (_I, [_I, _I, _I, _I, _I, _I, ctypes.POINTER(_I), ctypes.POINTER(_I)]),
    "pbb_plan_forward_query_tiles": (_I, [_I, _I, _I, _I, _I, _I]),
    "pbb_ring_from_sequence": (_I, [_P, _P, _I, _P, _P, _I, _I, _I, _I, _I, _P]),
    "pbb_backward": (_I, [_P, _P, _P, _P, _P, _P, _P, _P, _P, _P, _I, _I, _I, _I, _I, _I, _P]),
    "pbb_advance_positions": (_I, [_P, _I, _P]),
    "pbb_get_device_status": (_I, [_P]),
    "pbb_set_wait_timeout_ns": (_I, [_ULL]),
    "pbb_set_chunk_keys": (_I, [_I]),
    "pbb_set_kernel": (_I, [_I]),
    "pbb_plan_chunk_keys": (_I, [_I, _I, _I, _I, _I, _I]),
    "pbb_plan_kernel": (_I, [_I, _I, _I, _I, _I, _I]),
    "pbb_plan_support_order": (_I, [_I, _I, _I, _I, _I, _I, _I]),
    "pbb_stream_read": (_I, [_P, _SZ, _P, _P]),
    "pbb_error_string": (ctypes.c_char_p, [_I]),
}

_HERE = os.path.dirname(os.path.abspath(__file__))
lib_path = os.path.join(_HERE, "libpbb.so")
_lib = None
_lock = threading.Lock()


class PbbError(RuntimeError):
    def __init__(self, code: int, what: str = ""):
        self.code = code
        super().__init__(f"{what}: {error_string(code)} ({code})" if what else error_string(code))


def lib() -> ctypes.CDLL:
    """The loaded libpbb.so (raises if it has not been built)."""
    global _lib
    with _lock:
        if _lib is None:
            if not os.path.exists(lib_path):
                raise RuntimeError(f"libpbb.so not built at {lib_path}; run __graft_entry__.build()")
            handle = ctypes.CDLL(lib_path)
            for name, (res, args) in EXPORTS.items():
                fn = getattr(handle, name)
                fn.restype = res
                fn.argtypes = args
            _lib = handle
        return _lib


def error_string(code: int) -> str:
    try:
        return lib().pbb_error_string(code).decode()
    except Exception:  # noqa: BLE001 - library not loadable: still describe the code
        return f"pbb error {code}"


def _check(rc: int, what: str) -> None:
    if rc != PBB_OK:
        raise PbbError(rc, what)


def _dt(dtype: torch.dtype) -> int:
    if dtype == torch.bfloat16:
        return PBB_BF16
    if dtype == torch.float32:
        return PBB_F32
    raise TypeError(f"unsupported element type {dtype} (bf16 or fp32)")


def _stream(stream) -> ctypes.c_void_p:
    s = torch.cuda.current_stream() if stream is None else stream
    return ctypes.c_void_p(s.cuda_stream)


def _dev(t: torch.Tensor, name: str, dtype=None) -> int:
    if not isinstance(t, torch.Tensor) or not t.is_cuda:
        raise TypeError(f"{name} must be a CUDA tensor")
    if not t.is_contiguous():
        raise ValueError(f"{name} must be contiguous")
    if dtype is not None and t.dtype != dtype:
        raise TypeError(f"{name} must be {dtype}, got {t.dtype}")
    return t.data_ptr()


def ring_bytes(batch: int, Hkv: int, d: int, B: int, dtype: torch.dtype = torch.bfloat16) -> int:
    """Bytes of one ring (K or V); the pair is twice this (Appendix F.1)."""
    return int(lib().pbb_ring_bytes(batch, Hkv, d, B, _dt(dtype)))


class _CudaArray:
    """Minimal __cuda_array_interface__ view of library-owned device memory."""

    def __init__(self, ptr: int, shape, typestr: str):
        self.__cuda_array_interface__ = {"shape": tuple(shape), "typestr": typestr,
                                         "data": (ptr, False), "version": 3, "strides": None}


class Rings:
    """K and V rings allocated by pbb_ring_alloc; freed with ``free()`` or at collection."""

    def __init__(self, batch: int, Hkv: int, d: int, B: int, dtype=torch.bfloat16, stream=None):
        k, v = ctypes.c_void_p(), ctypes.c_void_p()
        self._stream = stream
        _check(lib().pbb_ring_alloc(ctypes.byref(k), ctypes.byref(v), batch, Hkv, d, B, _dt(dtype),
                                    _stream(stream)), "pbb_ring_alloc")
        self.k_ptr, self.v_ptr = k.value, v.value
        self.shape = (batch, Hkv, B, d)
        self.dtype = dtype
        typestr = "<i2" if dtype == torch.bfloat16 else "<f4"
        dev = torch.cuda.current_device()

        def view(ptr):
            t = torch.as_tensor(_CudaArray(ptr, self.shape, typestr), device=f"cuda:{dev}")
            return t.view(torch.bfloat16) if dtype == torch.bfloat16 else t

        self.k = view(self.k_ptr)
        self.v = view(self.v_ptr)

    def free(self) -> None:
        if getattr(self, "k_ptr", None):
            self.k = self.v = None
            _check(lib().pbb_ring_free(self.k_ptr, self.v_ptr, _stream(self._stream)), "pbb_ring_free")
            self.k_ptr = self.v_ptr = None

    def __del__(self):
        try:
            self.free()
        except Exception:  # noqa: BLE001 - interpreter shutdown
            pass


def ring_alloc(batch: int, Hkv: int, d: int, B: int, dtype=torch.bfloat16, stream=None) -> Rings:
    return Rings(batch, Hkv, d, B, dtype, stream)


def ring_prefill(k_hist: torch.Tensor, v_hist: torch.Tensor, pos: torch.Tensor,
                 k_ring: torch.Tensor, v_ring: torch.Tensor, stream=None) -> None:
    """Ring of sequences resuming at pos[b] from the B positions before it ([batch, Hkv, B, d])."""
    batch, Hkv, B, d = k_ring.shape
    dtype = k_ring.dtype
    for name, t in (("k_hist", k_hist), ("v_hist", v_hist), ("v_ring", v_ring)):
        if tuple(t.shape) != (batch, Hkv, B, d):
            raise ValueError(f"{name} must have shape {(batch, Hkv, B, d)}")
    if pos.numel() != batch:
        raise ValueError("pos must have batch entries")
    _check(lib().pbb_ring_prefill(_dev(k_hist, "k_hist", dtype), _dev(v_hist, "v_hist", dtype),
                                  _dev(pos, "pos", torch.int32), _dev(k_ring, "k_ring", dtype),
                                  _dev(v_ring, "v_ring", dtype), batch, Hkv, d, B, _dt(dtype),
                                  _stream(stream)), "pbb_ring_prefill")


def _step_shapes(q, k_new, v_new, k_ring, v_ring, pos, out):
    batch, Hq, d = q.shape
    _, Hkv, B, d2 = k_ring.shape
    dtype = q.dtype
    if d2 != d or k_ring.shape[0] != batch or tuple(v_ring.shape) != tuple(k_ring.shape):
        raise ValueError("ring shape must be [batch, Hkv, B, d]")
    if tuple(k_new.shape) != (batch, Hkv, d) or tuple(v_new.shape) != (batch, Hkv, d):
        raise ValueError("k_new/v_new must be [batch, Hkv, d]")
    if pos.numel() != batch:
        raise ValueError("pos must have batch entries")
    if out is None:
        out = torch.empty((batch, Hq, d), dtype=torch.float32, device=q.device)
    elif tuple(out.shape) != (batch, Hq, d):
        raise ValueError("out must be [batch, Hq, d]")
    return batch, Hq, Hkv, d, B, dtype, out


def decode_step(q: torch.Tensor, k_new: torch.Tensor, v_new: torch.Tensor, k_ring: torch.Tensor,
                v_ring: torch.Tensor, pos: torch.Tensor, out: torch.Tensor | None = None,
                stream=None) -> torch.Tensor:
    """One PBB decode step (include/pbb.h: pbb_decode_step / pbb_decode_step_f32).

    q [batch, Hq, d], k_new/v_new [batch, Hkv, d], rings [batch, Hkv, B, d] (bf16 or
    fp32, all the same), pos [batch] int32 on the device, out [batch, Hq, d] fp32.
    """
    batch, Hq, Hkv, d, B, dtype, out = _step_shapes(q, k_new, v_new, k_ring, v_ring, pos, out)
    fn = lib().pbb_decode_step if _dt(dtype) == PBB_BF16 else lib().pbb_decode_step_f32
    _check(fn(_dev(q, "q", dtype), _dev(k_new, "k_new", dtype), _dev(v_new, "v_new", dtype),
              _dev(k_ring, "k_ring", dtype), _dev(v_ring, "v_ring", dtype),
              _dev(pos, "pos", torch.int32), _dev(out, "out", torch.float32), batch, Hq, Hkv, d, B,
              _stream(stream)), "pbb_decode_step")
    return out


def decode_step_layers(q: torch.Tensor, k_new: torch.Tensor, v_new: torch.Tensor, k_ring: torch.Tensor,
                       v_ring: torch.Tensor, pos: torch.Tensor, out: torch.Tensor | None = None,
                       stream=None) -> torch.Tensor:
    """One decode step of L layers in one launch (pbb_decode_step_layers): q [L, batch, Hq, d],
    k_new/v_new [L, batch, Hkv, d], rings [L, batch, Hkv, B, d], pos [batch] shared by the layers,
    out [L, batch, Hq, d] fp32."""
    L, batch, Hq, d = q.shape
    _, _, Hkv, B, d2 = k_ring.shape
    dtype = q.dtype
    if d2 != d or tuple(k_ring.shape[:2]) != (L, batch) or tuple(v_ring.shape) != tuple(k_ring.shape):
        raise ValueError("rings must be [L, batch, Hkv, B, d]")
    if tuple(k_new.shape) != (L, batch, Hkv, d) or tuple(v_new.shape) != (L, batch, Hkv, d):
        raise ValueError("k_new/v_new must be [L, batch, Hkv, d]")
    if pos.numel() != batch:
        raise ValueError("pos must have batch entries")
    if out is None:
        out = torch.empty((L, batch, Hq, d), dtype=torch.float32, device=q.device)
    elif tuple(out.shape) != (L, batch, Hq, d):
        raise ValueError("out must be [L, batch, Hq, d]")
    _check(lib().pbb_decode_step_layers(_dev(q, "q", dtype), _dev(k_new, "k_new", dtype),
                                        _dev(v_new, "v_new", dtype), _dev(k_ring, "k_ring", dtype),
                                        _dev(v_ring, "v_ring", dtype), _dev(pos, "pos", torch.int32),
                                        _dev(out, "out", torch.float32), L, batch, Hq, Hkv, d, B, _dt(dtype),
                                        _stream(stream)), "pbb_decode_step_layers")
    return out


def swa_decode_step(q: torch.Tensor, k_new: torch.Tensor, v_new: torch.Tensor, k_ring: torch.Tensor,
                    v_ring: torch.Tensor, pos: torch.Tensor, out: torch.Tensor | None = None,
                    window: int | None = None, stream=None) -> torch.Tensor:
    """Sliding-window decode step over the same rings (pbb_swa_decode_step): the
    support is {t-w+1, ..., t}, w = window (default B). Arguments as ``decode_step``."""
    batch, Hq, Hkv, d, B, dtype, out = _step_shapes(q, k_new, v_new, k_ring, v_ring, pos, out)
    w = B if window is None else int(window)
    _check(lib().pbb_swa_decode_step(_dev(q, "q", dtype), _dev(k_new, "k_new", dtype),
                                     _dev(v_new, "v_new", dtype), _dev(k_ring, "k_ring", dtype),
                                     _dev(v_ring, "v_ring", dtype), _dev(pos, "pos", torch.int32),
                                     _dev(out, "out", torch.float32), batch, Hq, Hkv, d, B, w,
                                     _dt(dtype), _stream(stream)), "pbb_swa_decode_step")
    return out


class HostStep:
    """Device staging for ``decode_step_host`` (reused across calls of the same shape)."""

    def __init__(self, batch: int, Hq: int, Hkv: int, d: int, dtype, device):
        self.q = torch.empty((batch, Hq, d), dtype=dtype, device=device)
        self.k = torch.empty((batch, Hkv, d), dtype=dtype, device=device)
        self.v = torch.empty((batch, Hkv, d), dtype=dtype, device=device)
        self.out = torch.empty((batch, Hq, d), dtype=torch.float32, device=device)


def decode_step_host(q_h: torch.Tensor, k_h: torch.Tensor, v_h: torch.Tensor, k_ring: torch.Tensor,
                     v_ring: torch.Tensor, pos: torch.Tensor, out_h: torch.Tensor,
                     staging: HostStep, stream=None) -> None:
    """decode_step with the step's inputs and output in (pinned) host memory.

    Copies q/k/v host -> device, runs the step, copies out device -> host, all
    enqueued on the stream; the caller synchronises before reading out_h.
    """
    s = torch.cuda.current_stream() if stream is None else stream
    with torch.cuda.stream(s):
        staging.q.copy_(q_h, non_blocking=True)
        staging.k.copy_(k_h, non_blocking=True)
        staging.v.copy_(v_h, non_blocking=True)
        decode_step(staging.q, staging.k, staging.v, k_ring, v_ring, pos, staging.out, stream=s)
        out_h.copy_(staging.out, non_blocking=True)


class HostPipeline:
    """Decode steps whose inputs and outputs live in (pinned) host memory, with the
    transfers overlapped with the device work of neighbouring steps.

    Two device staging sets alternate between steps. Step i copies its q/k/v in on
    an input-copy stream while the compute stream may still run step i-1; the
    compute stream waits for those copies, runs the decode step and advances the
    positions; an output-copy stream then copies the output back. Events keep a
    staging set from being overwritten before its previous step is done with it.
    Call ``synchronize()`` before reading the host outputs.
    """

    def __init__(self, batch: int, Hq: int, Hkv: int, d: int, dtype, device, compute_stream=None,
                 window: int | None = None):
        self.window = window  # None: PBB steps; an integer: sliding-window steps of that window
        self.compute = torch.cuda.current_stream(device) if compute_stream is None else compute_stream
        self.copy_in = torch.cuda.Stream(device=device)
        self.copy_out = torch.cuda.Stream(device=device)
        self.sets = [HostStep(batch, Hq, Hkv, d, dtype, device) for _ in range(2)]
        self.inputs_ready = [torch.cuda.Event() for _ in range(2)]
        self.inputs_used = [torch.cuda.Event() for _ in range(2)]
        self.output_ready = [torch.cuda.Event() for _ in range(2)]
        self.output_sent = [torch.cuda.Event() for _ in range(2)]
        self.i = 0

    def step(self, q_h, k_h, v_h, k_ring, v_ring, pos, out_h) -> None:
        j = self.i % 2
        st = self.sets[j]
        if self.i >= 2:
            self.copy_in.wait_event(self.inputs_used[j])   # step i-2 has read these inputs
            self.compute.wait_event(self.output_sent[j])   # and its output has left this buffer
        with torch.cuda.stream(self.copy_in):
            st.q.copy_(q_h, non_blocking=True)
            st.k.copy_(k_h, non_blocking=True)
            st.v.copy_(v_h, non_blocking=True)
            self.inputs_ready[j].record(self.copy_in)
        self.compute.wait_event(self.inputs_ready[j])
        if self.window is None:
            decode_step(st.q, st.k, st.v, k_ring, v_ring, pos, st.out, stream=self.compute)
        else:
            swa_decode_step(st.q, st.k, st.v, k_ring, v_ring, pos, st.out, window=self.window,
                            stream=self.compute)
        self.inputs_used[j].record(self.compute)
        self.output_ready[j].record(self.compute)
        advance_positions(pos, stream=self.compute)
        self.copy_out.wait_event(self.output_ready[j])
        with torch.cuda.stream(self.copy_out):
            out_h.copy_(st.out, non_blocking=True)
            self.output_sent[j].record(self.copy_out)
        self.i += 1

    def last_output_event(self) -> torch.cuda.Event:
        """Event recorded after the output copy of the latest step."""
        return self.output_sent[(self.i - 1) % 2]

    def synchronize(self) -> None:
        self.copy_in.synchronize()
        self.compute.synchronize()
        self.copy_out.synchronize()


def forward(q: torch.Tensor, k: torch.Tensor, v: torch.Tensor, B: int, out: torch.Tensor | None = None,
            lse: torch.Tensor | bool | None = True, out_dtype=torch.bfloat16, stream=None):
    """PBB attention for every position of whole sequences (pbb_forward).

    q [batch, Hq, n, d], k/v [batch, Hkv, n, d] bf16 on the device; B the block size.
    Returns (out [batch, Hq, n, d] out_dtype, lse [batch, Hq, n] fp32 or None).
    lse: True allocates it, a tensor receives it, None/False skips it.
    """
    batch, Hq, n, d = q.shape
    Hkv = k.shape[1]
    if tuple(k.shape) != (batch, Hkv, n, d) or tuple(v.shape) != tuple(k.shape):
        raise ValueError("k/v must be [batch, Hkv, n, d] with q's batch, n and d")
    if out is None:
        out = torch.empty((batch, Hq, n, d), dtype=out_dtype, device=q.device)
    elif tuple(out.shape) != (batch, Hq, n, d):
        raise ValueError("out must be [batch, Hq, n, d]")
    if lse is True:
        lse = torch.empty((batch, Hq, n), dtype=torch.float32, device=q.device)
    elif lse is False:
        lse = None
    if lse is not None and tuple(lse.shape) != (batch, Hq, n):
        raise ValueError("lse must be [batch, Hq, n]")
    _check(lib().pbb_forward(_dev(q, "q", torch.bfloat16), _dev(k, "k", torch.bfloat16),
                             _dev(v, "v", torch.bfloat16), _dev(out, "out", out.dtype),
                             _dev(lse, "lse", torch.float32) if lse is not None else None,
                             batch, Hq, Hkv, n, d, B, _dt(out.dtype), _stream(stream)), "pbb_forward")
    return out, lse


def backward(q: torch.Tensor, k: torch.Tensor, v: torch.Tensor, out: torch.Tensor, dout: torch.Tensor,
             lse: torch.Tensor, B: int, stream=None, dq: torch.Tensor | None = None,
             dk: torch.Tensor | None = None, dv: torch.Tensor | None = None):
    """Gradients (dq, dk, dv), fp32, of pbb_forward (pbb_backward). out and lse are the
    forward's outputs for q, k, v; dout is the upstream gradient (bf16, shaped like out).
    dq, dk, dv: buffers to receive the gradients (allocated when None)."""
    batch, Hq, n, d = q.shape
    Hkv = k.shape[1]
    for name, t, shape in (("k", k, (batch, Hkv, n, d)), ("v", v, (batch, Hkv, n, d)),
                           ("out", out, (batch, Hq, n, d)), ("dout", dout, (batch, Hq, n, d)),
                           ("lse", lse, (batch, Hq, n))):
        if tuple(t.shape) != shape:
            raise ValueError(f"{name} must have shape {shape}")
    dev = q.device
    delta = torch.empty((batch, Hq, n), dtype=torch.float32, device=dev)
    grads = []
    for name, t, shape in (("dq", dq, (batch, Hq, n, d)), ("dk", dk, (batch, Hkv, n, d)),
                           ("dv", dv, (batch, Hkv, n, d))):
        if t is None:
            t = torch.empty(shape, dtype=torch.float32, device=dev)
        elif tuple(t.shape) != shape:
            raise ValueError(f"{name} must have shape {shape}")
        grads.append(t)
    dq, dk, dv = grads
    bf = torch.bfloat16
    _check(lib().pbb_backward(_dev(q, "q", bf), _dev(k, "k", bf), _dev(v, "v", bf), _dev(out, "out", bf),
                              _dev(dout, "dout", bf), _dev(lse, "lse", torch.float32),
                              _dev(delta, "delta", torch.float32), _dev(dq, "dq", torch.float32),
                              _dev(dk, "dk", torch.float32), _dev(dv, "dv", torch.float32), batch, Hq, Hkv, n, d,
                              B, _stream(stream)), "pbb_backward")
    return dq, dk, dv


def ring_from_sequence(k: torch.Tensor, v: torch.Tensor, k_ring: torch.Tensor, v_ring: torch.Tensor,
                       stream=None) -> None:
    """Rings [batch, Hkv, B, d] of sequences whose positions 0..n-1 are k/v [batch, Hkv, n, d]
    (pbb_ring_from_sequence); the next decode step is at position n."""
    batch, Hkv, B, d = k_ring.shape
    n = k.shape[2]
    dtype = k_ring.dtype
    if tuple(k.shape) != (batch, Hkv, n, d) or tuple(v.shape) != tuple(k.shape):
        raise ValueError("k/v must be [batch, Hkv, n, d] matching the rings")
    _check(lib().pbb_ring_from_sequence(_dev(k, "k", dtype), _dev(v, "v", dtype), n,
                                        _dev(k_ring, "k_ring", dtype), _dev(v_ring, "v_ring", dtype),
                                        batch, Hkv, d, B, _dt(dtype), _stream(stream)),
           "pbb_ring_from_sequence")


def advance_positions(pos: torch.Tensor, stream=None) -> None:
    """pos += 1 on the device."""
    _check(lib().pbb_advance_positions(_dev(pos, "pos", torch.int32), pos.numel(), _stream(stream)),
           "pbb_advance_positions")


def stream_read(buf: torch.Tensor, sink: torch.Tensor, stream=None) -> None:
    """Read every byte of the contiguous device tensor `buf` once (pbb_stream_read), xor-folded
    into the int64 device tensor `sink`: the read-only HBM bandwidth probe."""
    if not buf.is_cuda or not buf.is_contiguous() or not sink.is_cuda or sink.dtype != torch.int64:
        raise ValueError("buf must be a contiguous device tensor and sink an int64 device tensor")
    _check(lib().pbb_stream_read(ctypes.c_void_p(buf.data_ptr()), buf.numel() * buf.element_size(),
                                 ctypes.c_void_p(sink.data_ptr()), _stream(stream)), "pbb_stream_read")


def get_device_status(stream=None) -> int:
    """Synchronise and return (and clear) the device status word (PBB_OK or a PBB_ERR_DEVICE_* code)."""
    return int(lib().pbb_get_device_status(_stream(stream)))


def reserve_workspace(max_batch: int, Hq: int, Hkv: int, d: int, B: int, dtype=torch.bfloat16,
                      stream=None) -> None:
    """Grow the workspace of (current device, `stream`, default the current stream) for steps of
    this shape, e.g. on the stream a CUDA graph will be captured on."""
    _check(lib().pbb_reserve_workspace(max_batch, Hq, Hkv, d, B, _dt(dtype), _stream(stream)),
           "pbb_reserve_workspace")


def set_wait_timeout_ns(ns: int) -> None:
    _check(lib().pbb_set_wait_timeout_ns(int(ns)), "pbb_set_wait_timeout_ns")


def set_chunk_keys(keys: int) -> int:
    """Override the keys per CTA (0 = automatic); returns the previous setting."""
    prev = int(lib().pbb_set_chunk_keys(int(keys)))
    if prev < 0:
        raise PbbError(prev, "pbb_set_chunk_keys")
    return prev


def plan_chunk_keys(batch: int, Hq: int, Hkv: int, d: int, B: int, dtype=torch.bfloat16) -> int:
    return int(lib().pbb_plan_chunk_keys(batch, Hq, Hkv, d, B, _dt(dtype)))


PBB_KERNEL_AUTO = -1
PBB_KERNEL_CUDA_CORES = 0
PBB_KERNEL_TENSOR_CORES = 1
_KERNEL_NAMES = {"auto": PBB_KERNEL_AUTO, "cuda_cores": PBB_KERNEL_CUDA_CORES,
                 "tensor_cores": PBB_KERNEL_TENSOR_CORES}


def plan_forward(batch: int, Hq: int, Hkv: int, n: int, d: int, B: int) -> tuple:
    """(keys per K/V tile, persistent CTAs per SM) of pbb_forward for these sizes."""
    nk, ctas = _I(0), _I(0)
    _check(int(lib().pbb_plan_forward(batch, Hq, Hkv, n, d, B, ctypes.byref(nk), ctypes.byref(ctas))),
           "pbb_plan_forward")
    return nk.value, ctas.value


def set_kernel(kernel: str) -> str:
    """Kernel choice for later decode steps: 'auto' (default), 'cuda_cores', or
    'tensor_cores' (every step the tensor-core kernel supports, whatever the batch).
    Returns the previous choice."""
    if kernel not in _KERNEL_NAMES:
        raise ValueError(f"kernel must be one of {sorted(_KERNEL_NAMES)}")
    prev = int(lib().pbb_set_kernel(_KERNEL_NAMES[kernel]))
    if prev < PBB_KERNEL_AUTO:
        raise PbbError(prev, "pbb_set_kernel")
    return {v: k for k, v in _KERNEL_NAMES.items()}[prev]


def plan_forward_query_tiles(batch: int, Hq: int, Hkv: int, n: int, d: int, B: int) -> int:
    """Query tiles one CTA of pbb_forward works on at once for these sizes: 2 for the paired
    kernel, else 1 (pbb_plan_forward_query_tiles)."""
    rc = int(lib().pbb_plan_forward_query_tiles(batch, Hq, Hkv, n, d, B))
    if rc < 0:
        raise PbbError(rc, "pbb_plan_forward_query_tiles")
    return rc


def plan_support_order(batch: int, Hq: int, Hkv: int, d: int, B: int, window: int = 0,
                       dtype=torch.bfloat16) -> bool:
    """Whether a step of this shape first sorts its sequences by support length (one more kernel)."""
    rc = int(lib().pbb_plan_support_order(batch, Hq, Hkv, d, B, window, _dt(dtype)))
    if rc < 0:
        raise PbbError(rc, "pbb_plan_support_order")
    return rc == 1


def plan_kernel(batch: int, Hq: int, Hkv: int, d: int, B: int, dtype=torch.bfloat16) -> str:
    """'cuda_cores' or 'tensor_cores': the kernel a step of this shape runs."""
    rc = int(lib().pbb_plan_kernel(batch, Hq, Hkv, d, B, _dt(dtype)))
    if rc < 0:
        raise PbbError(rc, "pbb_plan_kernel")
    return "tensor_cores" if rc == PBB_KERNEL_TENSOR_CORES else "cuda_cores"
