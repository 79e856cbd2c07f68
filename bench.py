#!/usr/bin/env python3
"""Benchmark of the fused PBB decode step (ring append + attention over A(t)).

Default workload (the steady-state throughput point with the largest rings):
batch 512, Hq 32, Hkv 8, d 128, B 4096, bf16, every sequence at its own
position t0 ~ U[B, 2^20) so the phase r is random and the bridge exists.
Rings: 2 x 4.3 GB, far larger than L2, so every step streams from HBM.

A step is one pbb_decode_step over the whole batch plus the device-side
position advance. Prints one JSON line (rank 0):
  value      decode-core tokens*heads/s = batch * Hq * steps / time, summed over ranks
  roofline   algorithmic bytes per launch / mean kernel time vs measured HBM copy bandwidth
  e2e        the same metric through the host-memory entry (H2D of q/k/v, D2H of out per step)
  cpu_baseline  the fp64 oracle timed on the host cores on a bounded sample

--impl reference times the fp64 CPU oracle (the only reference this method has)
on a bounded sample per step. --sweep prints one line per throughput-sweep point.
--pattern swa times the sliding-window control (window B, same rings and
kernel family) instead, --pattern both prints the PBB line and then the
control's; the control lines carry their own metric name. --forward times the
whole-sequence forward (prefill) workloads, one line each, with a roofline
against HBM or the tensor cores, whichever bounds the workload; --backward
times the gradients (dq, dk, dv) on the same workloads.
"""
from __future__ import annotations

import argparse
import ctypes
import hashlib
import json
import os
import statistics
import subprocess
import sys
import threading
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

METRIC = "PBB decode-core tokens*heads/s"
METRIC_SWA = "SWA-B decode-core tokens*heads/s (control: window = B over the same ring)"
METRIC_FWD = "PBB forward tokens*heads/s"
METRIC_BWD = "PBB backward tokens*heads/s"
UNIT = "tokens*heads/s"
NOMINAL_HBM_GBS = 8000.0
FALLBACK_HBM_GBS = 6800.0
L2_BYTES = 129 * 1024 * 1024


def parse_args():
    ap = argparse.ArgumentParser(description=__doc__, formatter_class=argparse.RawDescriptionHelpFormatter)
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=400)
    ap.add_argument("--warmup", type=int, default=10)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--batch", type=int, default=512)
    ap.add_argument("--block", type=int, default=4096)
    ap.add_argument("--hq", type=int, default=0, help="query heads of the throughput point (default 32)")
    ap.add_argument("--hkv", type=int, default=0, help="KV heads of the throughput point (default 8)")
    ap.add_argument("--head-dim", type=int, default=0, help="head size of the throughput point (default 128)")
    ap.add_argument("--sweep", action="store_true", help="one line per throughput-sweep point")
    ap.add_argument("--workload", default="", help="a named workload of paper_2606_02680_gb300.inputs "
                    "(default: the throughput point given by --batch/--block)")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--cpu-seconds", type=float, default=12.0)
    ap.add_argument("--chunk", type=int, default=0, help="keys per CTA (0 = library plan)")
    ap.add_argument("--pattern", choices=["pbb", "swa", "both"], default="pbb",
                    help="attention pattern: PBB (default), the sliding-window control with window B, or both")
    ap.add_argument("--layers", type=int, default=1,
                    help="local layers per decode step (shared positions; their own rings and inputs)")
    ap.add_argument("--layer-launches", choices=["one", "each"], default="one",
                    help="with --layers > 1: one multi-layer launch per step, or one decode launch per layer")
    ap.add_argument("--forward", action="store_true",
                    help="time the whole-sequence forward (prefill) workloads instead of the decode step")
    ap.add_argument("--backward", action="store_true",
                    help="time the whole-sequence backward (dq, dk, dv) on the forward workloads")
    ap.add_argument("--fwd-workload", default="", help="one forward/backward workload (default: all)")
    ap.add_argument("--kernel", choices=["auto", "cuda_cores", "tensor_cores"], default="auto",
                    help="decode kernel choice (pbb_set_kernel); cuda_cores compares PBB and the window "
                         "control on the same kernel")
    ap.add_argument("--graph", choices=["auto", "on", "off"], default="auto",
                    help="replay the timed steps as one CUDA graph (auto: when a step is under 100 us, "
                         "where host launch overhead would otherwise dominate)")
    return ap.parse_args()


# ------------------------------------------------------------------ clocks --

_REASONS = {0x1: "gpu_idle", 0x2: "applications_clocks_setting", 0x4: "sw_power_cap",
            0x8: "hw_slowdown", 0x10: "sync_boost", 0x20: "sw_thermal_slowdown",
            0x40: "hw_thermal_slowdown", 0x80: "hw_power_brake_slowdown",
            0x100: "display_clock_setting"}


class ClockSampler:
    """Samples SM clock and clock-event reasons of one GPU through NVML (read only)."""

    def __init__(self, uuid: str | None, period_s: float = 0.001):
        self.period = period_s
        self.samples = []
        self.max_mhz = None
        self._stop = threading.Event()
        self._thread = None
        self._nvml = None
        self._h = None
        try:
            nv = ctypes.CDLL("libnvidia-ml.so.1")
            if nv.nvmlInit_v2() != 0:
                return
            h = ctypes.c_void_p()
            rc = -1
            if uuid:
                rc = nv.nvmlDeviceGetHandleByUUID(uuid.encode(), ctypes.byref(h))
            if rc != 0:
                idx = int(os.environ.get("CUDA_VISIBLE_DEVICES", "0").split(",")[0] or 0)
                rc = nv.nvmlDeviceGetHandleByIndex_v2(idx, ctypes.byref(h))
            if rc != 0:
                return
            self._nvml, self._h = nv, h
            mx = ctypes.c_uint()
            if nv.nvmlDeviceGetMaxClockInfo(h, 1, ctypes.byref(mx)) == 0:
                self.max_mhz = mx.value
        except OSError:
            pass

    def _run(self):
        nv, h = self._nvml, self._h
        clk, rs = ctypes.c_uint(), ctypes.c_ulonglong()
        get_reasons = getattr(nv, "nvmlDeviceGetCurrentClocksEventReasons", None) or \
            nv.nvmlDeviceGetCurrentClocksThrottleReasons
        while not self._stop.is_set():
            if nv.nvmlDeviceGetClockInfo(h, 1, ctypes.byref(clk)) == 0 and \
                    get_reasons(h, ctypes.byref(rs)) == 0:
                self.samples.append((clk.value, rs.value))
            time.sleep(self.period)

    def __enter__(self):
        if self._nvml is not None:
            self._thread = threading.Thread(target=self._run, daemon=True)
            self._thread.start()
        return self

    def __exit__(self, *exc):
        self._stop.set()
        if self._thread:
            self._thread.join()

    def summary(self):
        if not self.samples:
            return {"sm_mhz": None, "sm_max_mhz": self.max_mhz, "reasons": [], "samples": 0,
                    "source": "nvml unavailable" if self._nvml is None else "no samples"}
        reasons = set()
        for _, r in self.samples:
            for bit, name in _REASONS.items():
                if r & bit and name != "gpu_idle":
                    reasons.add(name)
        return {"sm_mhz": statistics.median(c for c, _ in self.samples), "sm_max_mhz": self.max_mhz,
                "reasons": sorted(reasons), "samples": len(self.samples), "source": "nvml"}


# ------------------------------------------------------------------- peaks --

def hbm_peak():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            return float(json.load(f)["hbm_gbs"]), "measured"
    except (OSError, KeyError, ValueError):
        return FALLBACK_HBM_GBS, "fallback"


def read_roof(dev, gib: int = 4, reps: int = 10):
    """Read-only HBM bandwidth on this GPU, now: pbb_stream_read over a `gib` GiB buffer (far
    larger than L2), best and median of `reps` event-timed launches after 3 warm-ups. A decode
    step reads its support and writes almost nothing, so this, not the copy bandwidth, is its
    ceiling; the copy figure stays the reported `peak`."""
    import torch

    import paper_2606_02680_gb300 as pbb

    nbytes = gib << 30
    buf = torch.empty(nbytes, dtype=torch.uint8, device=dev).random_(0, 256)
    sink = torch.zeros(1, dtype=torch.int64, device=dev)
    stream = torch.cuda.current_stream()
    for _ in range(3):
        pbb.stream_read(buf, sink)
    torch.cuda.synchronize()
    ev = [torch.cuda.Event(enable_timing=True) for _ in range(2 * reps)]
    for i in range(reps):
        ev[2 * i].record(stream)
        pbb.stream_read(buf, sink)
        ev[2 * i + 1].record(stream)
    torch.cuda.synchronize()
    if int(sink.item()) < 0:  # bit 63: a bounded wait on a copy ran out
        raise RuntimeError("pbb_stream_read: a wait on a bulk copy ran out")
    ms = [ev[2 * i].elapsed_time(ev[2 * i + 1]) for i in range(reps)]
    del buf
    torch.cuda.empty_cache()
    return {"gbs": nbytes / (min(ms) / 1e3) / 1e9, "gbs_median": nbytes / (statistics.median(ms) / 1e3) / 1e9,
            "how": f"pbb_stream_read over {gib} GiB (16 KiB bulk copies into shared memory, 8 in flight per "
                   f"SM, read once), best of {reps} event-timed launches in this run"}


def kernel_source_sha() -> str:
    """Hash of the decode kernel's source (the files the ncu traffic record depends on)."""
    h = hashlib.sha256()
    csrc = os.path.join(ROOT, "paper_2606_02680_gb300", "csrc")
    for name in ("pbb_decode.cu", "pbb_device.cuh", "pbb_internal.h"):
        with open(os.path.join(csrc, name), "rb") as f:
            h.update(name.encode() + b"\0" + f.read())
    return h.hexdigest()[:16]


def recorded_traffic(workload_key: str, launch_bytes: float):
    """DRAM traffic per launch from the committed ncu record, if it was taken on
    the current kernel source (else None). Scaled from the captured case by
    algorithmic bytes, which grow in proportion with the batch."""
    path = os.path.join(ROOT, "profiles", "traffic.json")
    try:
        with open(path) as f:
            rec = json.load(f)
    except (OSError, ValueError):
        return None
    entry = rec.get("workloads", {}).get(workload_key)
    if not entry or entry.get("kernel_source_sha") != kernel_source_sha():
        return None
    return entry["dram_bytes_per_launch"] / entry["algorithmic_bytes_per_launch"] * launch_bytes


# --------------------------------------------------------------- workload --

def describe(w):
    return (f"{w.name}: batch {w.batch}, Hq {w.Hq}, Hkv {w.Hkv}, d {w.d}, B {w.B}, {w.dtype}, "
            f"t0 ~ U[{w.t0_lo}, {w.t0_hi})")


def setup_device_workload(w, dev, pool: int, layers: int = 1):
    """Rings prefilled at each sequence's start position and a pool of step inputs. With
    layers > 1 every tensor holds layers x batch sequences (layer-major) that share the batch's
    positions; pos stays [batch]."""
    import torch

    import paper_2606_02680_gb300 as pbb
    from paper_2606_02680_gb300 import inputs

    t0 = inputs.start_positions(w)
    pos = t0.to(torch.int32).to(dev)
    dt = inputs.torch_dtype(w)
    wl = w.with_(batch=layers * w.batch)
    t_all = t0.repeat(layers)
    k_ring = torch.empty((wl.batch, w.Hkv, w.B, w.d), dtype=dt, device=dev)
    v_ring = torch.empty_like(k_ring)
    hk, hv = inputs.history_window(wl, t_all, device=dev)
    pbb.ring_prefill(hk, hv, t_all.to(torch.int32).to(dev), k_ring, v_ring)
    torch.cuda.synchronize()
    del hk, hv
    torch.cuda.empty_cache()
    steps_in = [inputs.step_inputs(wl, i, device=dev) for i in range(pool)]
    return t0, pos, k_ring, v_ring, steps_in


def stepper(window, layers=1, launches="one"):
    """The decode call of a step: PBB (window None) or the sliding window; with layers > 1 the
    tensors hold layers x batch sequences and the step is one multi-layer launch or one launch
    per layer."""
    import paper_2606_02680_gb300 as pbb

    if layers > 1:
        def multi(q, k, v, kr, vr, pos, out):
            L = layers
            sh = lambda x: x.view(L, x.shape[0] // L, *x.shape[1:])  # noqa: E731
            if launches == "one":
                pbb.decode_step_layers(sh(q), sh(k), sh(v), sh(kr), sh(vr), pos, sh(out))
            else:
                for l in range(L):
                    pbb.decode_step(sh(q)[l], sh(k)[l], sh(v)[l], sh(kr)[l], sh(vr)[l], pos, sh(out)[l])
        return multi
    if window is None:
        return pbb.decode_step
    return lambda q, k, v, kr, vr, pos, out: pbb.swa_decode_step(q, k, v, kr, vr, pos, out, window=window)


def time_device(w, dev, steps, warmup, dist=None, graph="auto", window=None, layers=1, launches="one"):
    """Device-timed loop; returns dict of timings.

    Eager mode records a CUDA event pair around every decode launch inside the
    timed region. Graph mode captures the `steps` steps once and times one
    replay (the protocol the paper uses for decode timing); the kernel's own
    duration then comes from an eager event-timed pass right after it.
    """
    import torch

    import paper_2606_02680_gb300 as pbb
    from paper_2606_02680_gb300 import bytemodel, inputs

    pool = 8
    decode = stepper(window, layers, launches)
    t0, pos, k_ring, v_ring, steps_in = setup_device_workload(w, dev, pool, layers)
    out = torch.empty((layers * w.batch, w.Hq, w.d), dtype=torch.float32, device=dev)
    pbb.reserve_workspace(layers * w.batch, w.Hq, w.Hkv, w.d, w.B, inputs.torch_dtype(w))
    stream = torch.cuda.current_stream()
    for i in range(warmup):
        q, k, v = steps_in[i % pool]
        decode(q, k, v, k_ring, v_ring, pos, out)
        pbb.advance_positions(pos)
    torch.cuda.synchronize()
    if graph == "auto":  # a short eager probe decides
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        for i in range(3):
            q, k, v = steps_in[i % pool]
            decode(q, k, v, k_ring, v_ring, pos, out)
            pbb.advance_positions(pos)
        e1.record(stream)
        torch.cuda.synchronize()
        warmup += 3
        graph = "on" if e0.elapsed_time(e1) / 3 < 0.1 else "off"
    use_graph = graph == "on"
    ev = [] if use_graph else [torch.cuda.Event(enable_timing=True) for _ in range(2 * steps)]
    start, end = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    g = None
    if use_graph:
        cap = torch.cuda.Stream(device=dev)
        # the steps captured on `cap` use that stream's workspace: size it before the capture
        pbb.reserve_workspace(layers * w.batch, w.Hq, w.Hkv, w.d, w.B, inputs.torch_dtype(w), stream=cap)
        cap.wait_stream(stream)
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=cap):
            for i in range(steps):
                q, k, v = steps_in[(warmup + i) % pool]
                decode(q, k, v, k_ring, v_ring, pos, out)
                pbb.advance_positions(pos)
        stream.wait_stream(cap)
        torch.cuda.synchronize()
    uuid = None
    try:
        uuid = "GPU-" + str(torch.cuda.get_device_properties(dev).uuid)
    except Exception:  # noqa: BLE001
        pass
    if dist is not None:
        dist.barrier()
    torch.cuda.synchronize()
    with ClockSampler(uuid) as clocks:
        start.record(stream)
        if use_graph:
            g.replay()
        else:
            for i in range(steps):
                q, k, v = steps_in[(warmup + i) % pool]
                ev[2 * i].record(stream)
                decode(q, k, v, k_ring, v_ring, pos, out)
                ev[2 * i + 1].record(stream)
                pbb.advance_positions(pos)
        end.record(stream)
        torch.cuda.synchronize()
    if dist is not None:
        dist.barrier()
    status = pbb.get_device_status()
    if status != pbb.PBB_OK:
        raise RuntimeError(f"device status {status} after the timed loop")
    total_ms = start.elapsed_time(end)
    t_np = t0.numpy()
    first = warmup
    if use_graph:
        # The launches of one step (decode and position advance) replay back to back, so the
        # replay's time per step bounds the decode kernel's duration from above. CUDA events
        # around single launches (eager, or recorded as nodes inside a graph) add the launch
        # latency of these short kernels and read longer than the whole step.
        kern_ms = [total_ms / steps] * steps
    else:
        kern_ms = [ev[2 * i].elapsed_time(ev[2 * i + 1]) for i in range(steps)]
    launch_bytes = [layers * bytemodel.step_bytes(t_np + first + i, w.Hq, w.Hkv, w.d, w.B, w.elem_bytes, window)
                    for i in range(steps)]
    res = {
        "total_ms": total_ms,
        "kernel_ms_mean": sum(kern_ms) / steps,
        "kernel_ms_median": statistics.median(kern_ms),
        "launch_bytes_mean": sum(launch_bytes) / steps,
        "clocks": clocks.summary(),
        "ring_bytes": 2 * k_ring.numel() * k_ring.element_size(),
        "timing": ("one CUDA-graph replay of the timed steps; the kernel duration in the roofline is the "
                   "replay's time per step (decode and position advance), an upper bound") if use_graph else
                  "eager launches; CUDA events around every decode launch",
        "state": (t0, pos, k_ring, v_ring, steps_in, out),
    }
    return res


def time_e2e(w, dev, steps, state, window=None):
    """Same steps through the host-memory API: every step copies its q/k/v in from
    pinned host memory and its output back, inside the timed region; the
    transfers of a step overlap the kernels of its neighbours (HostPipeline)."""
    import torch

    import paper_2606_02680_gb300 as pbb

    t0, pos, k_ring, v_ring, steps_in, _ = state
    pool = len(steps_in)
    host = [tuple(x.cpu().pin_memory() for x in s) for s in steps_in]
    out_h = [torch.empty((w.batch, w.Hq, w.d), dtype=torch.float32).pin_memory() for _ in range(4)]
    stream = torch.cuda.current_stream()
    pipe = pbb.HostPipeline(w.batch, w.Hq, w.Hkv, w.d, k_ring.dtype, dev, compute_stream=stream,
                            window=window)
    for i in range(3):
        q, k, v = host[i % pool]
        pipe.step(q, k, v, k_ring, v_ring, pos, out_h[i % 4])
    pipe.synchronize()
    start, end = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    torch.cuda.synchronize()
    start.record(stream)
    for i in range(steps):
        q, k, v = host[i % pool]
        pipe.step(q, k, v, k_ring, v_ring, pos, out_h[i % 4])
    stream.wait_event(pipe.last_output_event())  # the end event follows the last output copy
    end.record(stream)
    end.synchronize()
    ms = start.elapsed_time(end)
    q, k, v = host[0]
    h2d = sum(x.numel() * x.element_size() for x in (q, k, v))
    d2h = out_h[0].numel() * out_h[0].element_size()
    return {"value": w.batch * w.Hq * steps / (ms / 1e3), "unit": UNIT,
            "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h, "ms_per_step": ms / steps,
            "api": "paper_2606_02680_gb300.HostPipeline (pinned host q/k/v/out, copies overlapped)"}


def oracle_sample(w, seconds: float, seqs_per_call: int = 8, max_calls: int | None = None):
    """Time the fp64 oracle on sequences of workload w (inputs of the same recipe,
    generated on the host outside the timed region) until `seconds` have passed."""
    import oracle
    from paper_2606_02680_gb300 import inputs

    oracle.build()
    sub = w.with_(batch=seqs_per_call)
    t0 = inputs.start_positions(sub)
    hk, hv = inputs.history_window(sub, t0)
    q, k, v = inputs.step_inputs(sub, 0)
    hk = hk.clone()
    hv = hv.clone()
    # window of B+1 rows ending at the current token t0: rows t0-B .. t0
    import torch

    wk = torch.cat([hk, k.unsqueeze(2)], dim=2)[:, :, 1:]
    wv = torch.cat([hv, v.unsqueeze(2)], dim=2)[:, :, 1:]
    done = 0
    calls = 0
    elapsed = 0.0
    while True:  # at least one call
        t_start = time.perf_counter()
        oracle.attend(q, wk, wv, s0=(t0 - w.B + 1).numpy(), t=t0.numpy(), b=w.B)
        elapsed += time.perf_counter() - t_start
        done += seqs_per_call
        calls += 1
        if elapsed >= seconds or (max_calls is not None and calls >= max_calls):
            break
    return {"value": done * w.Hq / elapsed, "unit": UNIT, "cores": oracle.max_threads(),
            "kind": "oracle", "seconds": elapsed,
            "sample": f"{done} sequence-steps of {w.name} ({seqs_per_call} sequences per call, "
                      f"fp64 brute force over every position up to t)"}


# ------------------------------------------------------------------- arms --

def forward_flops_bytes(w):
    """Algorithmic FLOPs (4 d |A(t)| per query head and position: q.k and p.v, App. A.5)
    and bytes (q, k, v read once; bf16 out and fp32 lse written once) of one forward."""
    import numpy as np

    from paper_2606_02680_gb300 import bytemodel

    sizes = bytemodel.support_size(np.arange(w.n), w.B)
    flops = 4 * w.d * w.batch * w.Hq * int(sizes.sum())
    bytes_ = 2 * w.d * w.n * w.batch * (2 * w.Hq + 2 * w.Hkv) + 4 * w.batch * w.Hq * w.n
    return flops, bytes_


def backward_flops_bytes(w):
    """Algorithmic FLOPs of the backward: five products per (row, key) pair of a support
    (S, dP = dO.V, dV, dK, dQ), 10 d |A(t)| per query head and position; bytes: bf16 q, k,
    v, O, dO and fp32 lse read, fp32 dq, dk, dv written, the fp32 D row written and read."""
    import numpy as np

    from paper_2606_02680_gb300 import bytemodel

    sizes = bytemodel.support_size(np.arange(w.n), w.B)
    flops = 10 * w.d * w.batch * w.Hq * int(sizes.sum())
    rows_q, rows_k = w.batch * w.Hq * w.n, w.batch * w.Hkv * w.n
    bytes_ = (2 * w.d * (3 * rows_q + 2 * rows_k) + 4 * rows_q        # q, O, dO, k, v, lse
              + 4 * w.d * (rows_q + 2 * rows_k) + 8 * rows_q)         # dq, dk, dv, D
    return flops, bytes_


def tensor_peak():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            return float(json.load(f)["bf16_tflops"]), "measured (cuBLAS bf16 burst)"
    except (OSError, KeyError, ValueError):
        return 1900.0, "fallback"


def time_forward(w, dev, steps, warmup, dist=None):
    """Eager forward launches with CUDA events around each; inputs resident in HBM."""
    import torch

    import paper_2606_02680_gb300 as pbb
    from paper_2606_02680_gb300 import inputs

    q, k, v = inputs.sequence_inputs(w, device=dev)
    out = torch.empty((w.batch, w.Hq, w.n, w.d), dtype=torch.bfloat16, device=dev)
    lse = torch.empty((w.batch, w.Hq, w.n), dtype=torch.float32, device=dev)
    stream = torch.cuda.current_stream()
    for _ in range(warmup):
        pbb.forward(q, k, v, w.B, out=out, lse=lse)
    torch.cuda.synchronize()
    ev = [torch.cuda.Event(enable_timing=True) for _ in range(2 * steps)]
    start, end = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    uuid = None
    try:
        uuid = "GPU-" + str(torch.cuda.get_device_properties(dev).uuid)
    except Exception:  # noqa: BLE001
        pass
    if dist is not None:
        dist.barrier()
    torch.cuda.synchronize()
    with ClockSampler(uuid) as clocks:
        start.record(stream)
        for i in range(steps):
            ev[2 * i].record(stream)
            pbb.forward(q, k, v, w.B, out=out, lse=lse)
            ev[2 * i + 1].record(stream)
        end.record(stream)
        torch.cuda.synchronize()
    if dist is not None:
        dist.barrier()
    if pbb.get_device_status() != pbb.PBB_OK:
        raise RuntimeError("device status after the timed forward loop")
    kern = [ev[2 * i].elapsed_time(ev[2 * i + 1]) for i in range(steps)]
    return {"total_ms": start.elapsed_time(end), "kernel_ms_mean": sum(kern) / steps,
            "kernel_ms_median": statistics.median(kern), "clocks": clocks.summary(),
            "state": (q, k, v, out, lse)}


def time_forward_e2e(w, dev, steps, state):
    """Through the public API with host-resident inputs: each step copies q/k/v in from
    pinned host memory, runs the forward and copies out/lse back (all on one stream)."""
    import torch

    import paper_2606_02680_gb300 as pbb

    q, k, v, out, lse = state
    hq, hk, hv = (x.cpu().pin_memory() for x in (q, k, v))
    ho = torch.empty(out.shape, dtype=out.dtype).pin_memory()
    hl = torch.empty(lse.shape, dtype=lse.dtype).pin_memory()
    stream = torch.cuda.current_stream()

    def step():
        q.copy_(hq, non_blocking=True)
        k.copy_(hk, non_blocking=True)
        v.copy_(hv, non_blocking=True)
        pbb.forward(q, k, v, w.B, out=out, lse=lse)
        ho.copy_(out, non_blocking=True)
        hl.copy_(lse, non_blocking=True)

    step()
    torch.cuda.synchronize()
    start, end = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    start.record(stream)
    for _ in range(steps):
        step()
    end.record(stream)
    end.synchronize()
    ms = start.elapsed_time(end)
    return {"value": w.batch * w.Hq * w.n * steps / (ms / 1e3), "unit": UNIT,
            "h2d_bytes_per_step": sum(x.numel() * x.element_size() for x in (hq, hk, hv)),
            "d2h_bytes_per_step": ho.numel() * ho.element_size() + hl.numel() * hl.element_size(),
            "ms_per_step": ms / steps,
            "api": "paper_2606_02680_gb300.forward (pinned host q/k/v in, out/lse back, one stream)"}


def time_backward(w, dev, steps, warmup, dist=None):
    """Eager backward calls (three kernels each) with CUDA events around each; inputs resident."""
    import torch

    import paper_2606_02680_gb300 as pbb
    from paper_2606_02680_gb300 import inputs

    q, k, v = inputs.sequence_inputs(w, device=dev)
    g = torch.Generator(device=dev)
    g.manual_seed(w.seed + 1000)
    do = torch.randn((w.batch, w.Hq, w.n, w.d), generator=g, device=dev).to(torch.bfloat16)
    out, lse = pbb.forward(q, k, v, w.B)
    stream = torch.cuda.current_stream()
    for _ in range(warmup):
        pbb.backward(q, k, v, out, do, lse, w.B)
    torch.cuda.synchronize()
    ev = [torch.cuda.Event(enable_timing=True) for _ in range(2 * steps)]
    start, end = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    uuid = None
    try:
        uuid = "GPU-" + str(torch.cuda.get_device_properties(dev).uuid)
    except Exception:  # noqa: BLE001
        pass
    if dist is not None:
        dist.barrier()
    torch.cuda.synchronize()
    with ClockSampler(uuid) as clocks:
        start.record(stream)
        for i in range(steps):
            ev[2 * i].record(stream)
            pbb.backward(q, k, v, out, do, lse, w.B)
            ev[2 * i + 1].record(stream)
        end.record(stream)
        torch.cuda.synchronize()
    if dist is not None:
        dist.barrier()
    if pbb.get_device_status() != pbb.PBB_OK:
        raise RuntimeError("device status after the timed backward loop")
    kern = [ev[2 * i].elapsed_time(ev[2 * i + 1]) for i in range(steps)]
    return {"total_ms": start.elapsed_time(end), "kernel_ms_mean": sum(kern) / steps,
            "kernel_ms_median": statistics.median(kern), "clocks": clocks.summary(),
            "state": (q, k, v, out, do, lse)}


def time_backward_e2e(w, dev, steps, state):
    """The backward through the public API with host-resident tensors: q, k, v, O, dO, lse
    copied in from pinned host memory and dq, dk, dv copied back, every step, one stream."""
    import torch

    import paper_2606_02680_gb300 as pbb

    dev_t = state
    host = [x.cpu().pin_memory() for x in dev_t]
    stream = torch.cuda.current_stream()
    outs = None

    def step():
        nonlocal outs
        for d_, h_ in zip(dev_t, host):
            d_.copy_(h_, non_blocking=True)
        q, k, v, out, do, lse = dev_t
        dq, dk, dv = pbb.backward(q, k, v, out, do, lse, w.B)
        if outs is None:
            outs = [torch.empty(x.shape, dtype=x.dtype).pin_memory() for x in (dq, dk, dv)]
        for h_, d_ in zip(outs, (dq, dk, dv)):
            h_.copy_(d_, non_blocking=True)

    step()
    torch.cuda.synchronize()
    start, end = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    start.record(stream)
    for _ in range(steps):
        step()
    end.record(stream)
    end.synchronize()
    ms = start.elapsed_time(end)
    return {"value": w.batch * w.Hq * w.n * steps / (ms / 1e3), "unit": UNIT,
            "h2d_bytes_per_step": sum(x.numel() * x.element_size() for x in host),
            "d2h_bytes_per_step": sum(x.numel() * x.element_size() for x in outs),
            "ms_per_step": ms / steps,
            "api": "paper_2606_02680_gb300.backward (pinned host q/k/v/O/dO/lse in, dq/dk/dv back, one stream)"}


def oracle_backward_sample(w, seconds: float):
    """The fp64 oracle backward on a prefix of one (sequence, KV head) slice of the workload,
    grown until about `seconds` of CPU time; rows = positions x query heads of the prefix."""
    import torch

    import oracle
    from paper_2606_02680_gb300 import inputs

    oracle.build()
    n = min(w.n, 2 * w.B)
    done, elapsed = 0, 0.0
    while True:
        sub = w.with_(batch=1, Hq=w.group, Hkv=1, n=n)
        q, k, v = inputs.sequence_inputs(sub)
        do = torch.randn(q.shape, generator=torch.Generator().manual_seed(1)).to(torch.bfloat16)
        t_start = time.perf_counter()
        oracle.backward(q, k, v, do, w.B)
        elapsed += time.perf_counter() - t_start
        done += sub.Hq * n
        if elapsed >= seconds:
            break
    return {"value": done / elapsed, "unit": UNIT, "cores": oracle.max_threads(), "kind": "oracle",
            "seconds": elapsed,
            "sample": f"{done} (position, query head) rows of {w.name}: repeated backward passes over the "
                      f"first {n} positions of one sequence and KV head (fp64 chain rule, one thread per "
                      f"(sequence, KV head), so a single slice runs on one core)"}


def oracle_forward_sample(w, seconds: float, rows_per_call: int = 64):
    """The fp64 oracle forward on sampled rows of the workload (one sequence, one KV head)."""
    import numpy as np

    import oracle
    from paper_2606_02680_gb300 import inputs

    oracle.build()
    sub = w.with_(batch=1, Hq=w.group, Hkv=1)
    q, k, v = inputs.sequence_inputs(sub)
    rng = np.random.default_rng(0)
    done, elapsed = 0, 0.0
    while True:
        rows = np.stack([np.zeros(rows_per_call, dtype=np.int64), rng.integers(0, sub.Hq, rows_per_call),
                         rng.integers(0, w.n, rows_per_call)], axis=1)
        t_start = time.perf_counter()
        oracle.forward(q, k, v, w.B, rows=rows)
        elapsed += time.perf_counter() - t_start
        done += rows_per_call
        if elapsed >= seconds:
            break
    return {"value": done / elapsed, "unit": UNIT, "cores": oracle.max_threads(), "kind": "oracle",
            "seconds": elapsed,
            "sample": f"{done} output rows (position, head) of {w.name}, uniform positions, fp64 brute "
                      f"force over every position up to t (includes widening the slice to fp64)"}


def fwd_kernel_label(w):
    """The forward kernel a workload runs, with its launch shape."""
    import paper_2606_02680_gb300 as pbb

    nk, ctas = pbb.plan_forward(w.batch, w.Hq, w.Hkv, w.n, w.d, w.B)
    if pbb.plan_forward_query_tiles(w.batch, w.Hq, w.Hkv, w.n, w.d, w.B) == 2:
        return "forward_pair_kernel<%d,%d,%d keys,2 query tiles per CTA>" % (w.d, w.group, nk)
    return "forward_kernel<%d,%d,%d keys,%d CTAs/SM>" % (w.d, w.group, nk, ctas)


def run_forward(args, dist, rank, world, dev):
    import torch

    import paper_2606_02680_gb300 as pbb
    from paper_2606_02680_gb300 import inputs

    names = [args.fwd_workload] if args.fwd_workload else list(inputs.FORWARD_WORKLOADS)
    hbm, hbm_kind = hbm_peak()
    tpk, tpk_kind = tensor_peak()
    bwd = args.backward
    for name in names:
        w = inputs.FORWARD_WORKLOADS[name]
        w = w.with_(batch=shard_batch(w.batch, rank, world))
        res = (time_backward if bwd else time_forward)(w, dev, args.steps, args.warmup, dist)
        total_s = max_over_ranks(dist, res["total_ms"] / 1e3)
        units = sum_over_ranks(dist, w.batch * w.Hq * w.n * args.steps)
        flops, bytes_ = (backward_flops_bytes if bwd else forward_flops_bytes)(w)
        kern_s = res["kernel_ms_mean"] / 1e3
        t_hbm, t_tc = bytes_ / (hbm * 1e9), flops / (tpk * 1e12)
        if t_tc >= t_hbm:
            roof = {"bound": "tensor", "achieved": flops / kern_s / 1e12, "peak": tpk, "unit": "TFLOP/s",
                    "peak_kind": tpk_kind}
        else:
            roof = {"bound": "hbm", "achieved": bytes_ / kern_s / 1e9, "peak": hbm, "unit": "GB/s",
                    "peak_kind": hbm_kind}
        roof["frac"] = roof["achieved"] / roof["peak"]
        roof.update({"traffic": None,
                     "kernel": ("bwd_kv_tc_kernel<%d,%d> + bwd_q_tc_kernel<%d,%d> + delta_kernel<%d> (one call)"
                                % (w.d, w.group, w.d, w.group, w.d)) if bwd else
                               fwd_kernel_label(w),
                     "algorithmic_flops_per_launch": flops, "algorithmic_bytes_per_launch": bytes_,
                     "hbm_gbs": bytes_ / kern_s / 1e9, "tflops": flops / kern_s / 1e12,
                     "kernel_ms_mean": res["kernel_ms_mean"], "kernel_ms_median": res["kernel_ms_median"]})
        line = {
            "metric": METRIC_BWD if bwd else METRIC_FWD, "value": units / total_s, "unit": UNIT, "n_gpus": world,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": total_s * 1e3 / args.steps,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "bf16",
            "data": "synthetic (seeded N(0,1) q/k/v)",
            "config": {"workload": f"{w.name}: batch {w.batch}, Hq {w.Hq}, Hkv {w.Hkv}, d {w.d}, B {w.B}, n {w.n}, "
                                   + ("bf16 q/k/v/O/dO + fp32 lse in, fp32 dq/dk/dv out" if bwd else "bf16 out + fp32 lse"),
                       "batch_per_gpu": w.batch, "Hq": w.Hq, "Hkv": w.Hkv, "head_dim": w.d, "block": w.B,
                       "n": w.n, "l2": "inputs larger than L2: q/k/v/out %.2f GB" % (bytes_ / 1e9),
                       "parallelism": f"dp{world} (independent sequences, no collective)"},
            "roofline": roof, "clocks": res["clocks"],
            "timing": "eager calls; CUDA events around every " + ("backward call (3 launches)" if bwd else
                                                                      "forward launch"),
            "gpu_launches": (3 if bwd else 1) * args.steps,
        }
        if not args.no_e2e:
            line["e2e"] = (time_backward_e2e if bwd else time_forward_e2e)(w, dev, min(args.steps, 10), res["state"])
        res.pop("state")
        torch.cuda.empty_cache()
        if rank == 0 and world == 1 and not args.no_cpu_baseline:
            line["cpu_baseline"] = (oracle_backward_sample if bwd else oracle_forward_sample)(w, args.cpu_seconds)
        if rank == 0:
            print(json.dumps(line), flush=True)


def dist_setup():
    world = int(os.environ.get("WORLD_SIZE", "1"))
    if world <= 1:
        return None, 0, 1, 0
    import torch
    import torch.distributed as dist

    rank = int(os.environ["RANK"])
    local = int(os.environ.get("LOCAL_RANK", rank))
    backend = "nccl" if torch.cuda.is_available() else "gloo"
    if torch.cuda.is_available():
        torch.cuda.set_device(local)
    dist.init_process_group(backend=backend)
    return dist, rank, world, local


def shard_batch(batch: int, rank: int, world: int, scaling: str = "weak"):
    """Sequences of one rank: weak scaling keeps `batch` per rank; strong splits it."""
    if scaling == "weak":
        return batch
    base, rem = divmod(batch, world)
    return base + (1 if rank < rem else 0)


def max_over_ranks(dist, x: float) -> float:
    if dist is None:
        return x
    import torch

    dev = torch.device("cuda", torch.cuda.current_device()) if torch.cuda.is_available() else "cpu"
    t = torch.tensor([x], dtype=torch.float64, device=dev)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def sum_over_ranks(dist, x: float) -> float:
    if dist is None:
        return x
    import torch

    dev = torch.device("cuda", torch.cuda.current_device()) if torch.cuda.is_available() else "cpu"
    t = torch.tensor([x], dtype=torch.float64, device=dev)
    dist.all_reduce(t, op=dist.ReduceOp.SUM)
    return float(t.item())


def run_ours(args):
    import torch

    import paper_2606_02680_gb300 as pbb
    from paper_2606_02680_gb300 import build as nvbuild
    from paper_2606_02680_gb300 import inputs

    dist, rank, world, local = dist_setup()
    if not torch.cuda.is_available():
        raise SystemExit("bench.py needs a GPU (no CPU fallback)")
    if rank == 0 or dist is None:
        nvbuild.build()
    if dist is not None:
        dist.barrier()
    dev = torch.device("cuda", local if dist is not None else 0)
    torch.cuda.set_device(dev)
    pbb.set_chunk_keys(args.chunk)
    pbb.set_kernel(args.kernel)

    if args.forward or args.backward:
        run_forward(args, dist, rank, world, dev)
        if dist is not None:
            dist.barrier()
            dist.destroy_process_group()
        return
    if args.workload:
        base = inputs.WORKLOADS[args.workload]
        points = [base.with_(batch=shard_batch(base.batch, rank, world))]
    elif args.sweep:
        points = [inputs.sweep_workload(shard_batch(b, rank, world), B)
                  for b in inputs.SWEEP_BATCHES for B in inputs.SWEEP_BLOCKS]
    else:
        w0 = inputs.sweep_workload(shard_batch(args.batch, rank, world), args.block)
        if args.hq or args.hkv or args.head_dim:
            hq, hkv, hd = args.hq or w0.Hq, args.hkv or w0.Hkv, args.head_dim or w0.d
            w0 = w0.with_(Hq=hq, Hkv=hkv, d=hd, name=f"{w0.name}_Hq{hq}_Hkv{hkv}" + (f"_d{hd}" if hd != w0.d else ""))
        points = [w0]
    peak, peak_kind = hbm_peak()
    patterns = {"pbb": ["pbb"], "swa": ["swa"], "both": ["pbb", "swa"]}[args.pattern]
    for w, pattern in [(w, p) for w in points for p in patterns]:
        window = w.B if pattern == "swa" else None
        res = time_device(w, dev, args.steps, args.warmup, dist, args.graph, window, args.layers,
                          args.layer_launches)
        total_s = max_over_ranks(dist, res["total_ms"] / 1e3)
        units = sum_over_ranks(dist, args.layers * w.batch * w.Hq * args.steps)
        value = units / total_s
        achieved = res["launch_bytes_mean"] / (res["kernel_ms_mean"] / 1e3) / 1e9
        key = w.name if window is None else f"{w.name}_swa"
        traffic = recorded_traffic(key, res["launch_bytes_mean"])
        # window steps follow the same kernel choice as PBB steps of the shape
        kernel = ("decode_kernel_tc<%d>" % w.d
                  if pbb.plan_kernel(w.batch, w.Hq, w.Hkv, w.d, w.B, inputs.torch_dtype(w)) == "tensor_cores"
                  else "decode_kernel<%d,%d,%d>" % (w.elem_bytes, w.d, w.group))
        # a decode call of this batch sorts its sequences by support length first (one more launch)
        call_batch = w.batch * (args.layers if args.layer_launches == "one" else 1)
        ordered = int(pbb.plan_support_order(call_batch, w.Hq, w.Hkv, w.d, w.B, window or 0, inputs.torch_dtype(w)))
        if ordered:
            kernel += " after support_order_kernel"
        line = {
            "metric": METRIC if window is None else METRIC_SWA, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": total_s * 1e3 / args.steps,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": w.dtype,
            "data": "synthetic (seeded N(0,1) K/V/q; rings prefilled consistent with each t0)",
            "config": {"workload": describe(w), "batch_per_gpu": w.batch, "Hq": w.Hq, "Hkv": w.Hkv,
                       "head_dim": w.d, "block": w.B,
                       "keys_per_cta": pbb.plan_chunk_keys(w.batch, w.Hq, w.Hkv, w.d, w.B),
                       "l2": ("inputs larger than L2: rings %.2f GB" % (res["ring_bytes"] / 1e9))
                       if res["ring_bytes"] > L2_BYTES else
                       "rings fit in L2 (%.1f MB): latency/L2-bound point, not an HBM claim" % (res["ring_bytes"] / 1e6),
                       "parallelism": f"dp{world} (independent sequences, no collective)"},
            "hbm_gbs": achieved,
            "frac_of_8tbs": achieved / NOMINAL_HBM_GBS,
            "roofline": {"bound": "hbm", "achieved": achieved, "peak": peak, "unit": "GB/s",
                         "frac": achieved / peak, "traffic": traffic,
                         "kernel": kernel,
                         "peak_kind": peak_kind + " copy bandwidth (read + write)",
                         "algorithmic_bytes_per_launch": res["launch_bytes_mean"],
                         "kernel_ms_mean": res["kernel_ms_mean"],
                         "kernel_ms_median": res["kernel_ms_median"]},
            "clocks": res["clocks"],
            "timing": res["timing"],
            "gpu_launches": (2 + ordered) * args.steps,
        }
        if not args.sweep and args.layers == 1 and w.batch * w.Hkv * w.B * w.d * w.elem_bytes * 2 > L2_BYTES:
            rr = read_roof(dev)
            line["roofline"]["read_roof"] = dict(rr, frac=achieved / rr["gbs"])
        if not args.no_e2e and not args.sweep and args.layers == 1:
            line["e2e"] = time_e2e(w, dev, args.steps, res["state"], window)
        res.pop("state")
        torch.cuda.empty_cache()
        if window is not None:
            line["config"]["window"] = window
        if args.layers > 1:
            line["config"]["layers"] = args.layers
            line["config"]["layer_launches"] = ("one multi-layer launch per step" if args.layer_launches == "one"
                                                else "one decode launch per layer")
            line["gpu_launches"] = ((2 + ordered) if args.layer_launches == "one"
                                    else args.layers * (1 + ordered) + 1) * args.steps
        if rank == 0 and world == 1 and not args.no_cpu_baseline and not args.sweep and window is None and \
                args.layers == 1:
            line["cpu_baseline"] = oracle_sample(w, args.cpu_seconds)
        if rank == 0:
            print(json.dumps(line), flush=True)
    if dist is not None:
        dist.barrier()
        dist.destroy_process_group()


def run_reference(args):
    """The fp64 oracle on the host cores; each step is a bounded sample of the workload."""
    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    if rank != 0:
        return
    from paper_2606_02680_gb300 import inputs

    w = inputs.sweep_workload(args.batch, args.block)
    seqs = 4
    for _ in range(args.warmup):
        oracle_sample(w, 0.0, seqs_per_call=seqs, max_calls=1)
    times = []
    for _ in range(args.steps):
        s = oracle_sample(w, 0.0, seqs_per_call=seqs, max_calls=1)
        times.append(s["seconds"])
        cores = s["cores"]
    total = sum(times)
    value = seqs * w.Hq * args.steps / total
    sample = (f"each step: {seqs} sequences of {w.name} (fp64 brute force over every "
              f"position up to t), not the whole batch")
    line = {
        "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": total * 1e3 / args.steps, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "config": {"workload": describe(w), "batch_per_gpu": w.batch, "Hq": w.Hq, "Hkv": w.Hkv,
                   "head_dim": w.d, "block": w.B},
        "impl": "reference",
        "cpu_baseline": {"value": value, "unit": UNIT, "cores": cores, "kind": "oracle",
                         "sample": sample},
        "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
        "gpu_launches": 0,
    }
    print(json.dumps(line), flush=True)


def main():
    args = parse_args()
    if args.impl == "reference":
        run_reference(args)
    else:
        run_ours(args)


if __name__ == "__main__":
    main()
