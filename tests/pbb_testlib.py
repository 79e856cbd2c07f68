"""Helpers shared by the GPU parity tests (test infrastructure).

The CUDA path is reached only through the binding (C ABI); expected values
come only from the oracle. Nothing here computes the method's arithmetic.
"""
from __future__ import annotations

import numpy as np
import torch

import oracle
import paper_2606_02680_gb300 as pbb
from paper_2606_02680_gb300 import inputs

# Accuracy bounds: bf16 inputs 1e-2, fp32 inputs 1e-5, on max |out - oracle| and
# on max |out - oracle| / max(|oracle|, 1) (fp32 output in both cases).
TOL = {"bf16": 1e-2, "f32": 1e-5}


def check_close(out, ref, dtype: str, what: str = "") -> float:
    out = np.asarray(out, dtype=np.float64)
    ref = np.asarray(ref, dtype=np.float64)
    assert out.shape == ref.shape, (out.shape, ref.shape)
    assert np.all(np.isfinite(out)), f"{what}: non-finite output"
    err = np.abs(out - ref)
    tol = TOL[dtype]
    mx = float(err.max()) if err.size else 0.0
    rel = float((err / np.maximum(np.abs(ref), 1.0)).max()) if err.size else 0.0
    assert mx <= tol and rel <= tol, f"{what}: max abs {mx:.3e}, max rel {rel:.3e} > {tol}"
    return mx


def ring_bytes_np(t: torch.Tensor) -> np.ndarray:
    """Device ring [batch, Hkv, B, d] -> uint8 [batch, Hkv, B, row_bytes] (exact bits)."""
    t = t.detach().cpu().contiguous()
    iv = t.view(torch.int16) if t.dtype == torch.bfloat16 else t.view(torch.int32)
    return iv.numpy().view(np.uint8).reshape(*t.shape[:-1], -1)


def _decode(q, k, v, k_ring, v_ring, pos, window):
    """PBB step (window None) or sliding-window step of `window` positions."""
    if window is None:
        return pbb.decode_step(q, k, v, k_ring, v_ring, pos)
    return pbb.swa_decode_step(q, k, v, k_ring, v_ring, pos, window=window)


def _expected(q, hk, hv, t, B, window):
    """Oracle output over history rows of positions t-B .. t (PBB or window)."""
    if window is None:
        return oracle.attend(q, hk, hv, s0=t - B, t=t, b=B)
    return oracle.attend_window(q, hk, hv, s0=t - B, t=t, w=window)


class SequentialRun:
    """Drive the GPU decode step over consecutive steps of a workload and keep the
    host copy of the history the oracle needs (start window + every new token).
    window=None runs PBB steps, an integer runs sliding-window steps of that
    window; ``step(window=...)`` overrides it for one step."""

    def __init__(self, w: inputs.Workload, device="cuda", prefill: bool = True, gen_device="cpu",
                 window=None):
        self.w = w
        self.window = window
        self.last_window = window
        self.dev = torch.device(device)
        self.dtype = inputs.torch_dtype(w)
        self.t0 = inputs.start_positions(w)
        self.pos = self.t0.to(torch.int32).to(self.dev)
        self.k_ring = torch.zeros((w.batch, w.Hkv, w.B, w.d), dtype=self.dtype, device=self.dev)
        self.v_ring = torch.zeros_like(self.k_ring)
        self.sim = oracle.RingSim(w.batch, w.Hkv, w.d, w.B, w.elem_bytes)
        # history rows: window (positions t0-B .. t0-1) then one row per step
        self.hk = torch.zeros((w.batch, w.Hkv, w.B + w.steps, w.d), dtype=self.dtype)
        self.hv = torch.zeros_like(self.hk)
        if prefill and int(self.t0.max()) > 0:
            wk, wv = inputs.history_window(w, self.t0, device=gen_device)
            self.hk[:, :, :w.B] = wk.cpu()
            self.hv[:, :, :w.B] = wv.cpu()
            pbb.ring_prefill(wk.to(self.dev), wv.to(self.dev), self.pos, self.k_ring, self.v_ring)
            self.sim.replay(self.hk[:, :, :w.B], self.hv[:, :, :w.B], (self.t0 - w.B).numpy())
        self.step_i = 0
        self.q_last = None

    def step(self, gen_device="cpu", window="default"):
        w, i = self.w, self.step_i
        win = self.window if window == "default" else window
        q, k, v = inputs.step_inputs(w, i, device=gen_device)
        q, k, v = q.cpu(), k.cpu(), v.cpu()
        self.hk[:, :, w.B + i] = k
        self.hv[:, :, w.B + i] = v
        out = _decode(q.to(self.dev), k.to(self.dev), v.to(self.dev), self.k_ring, self.v_ring,
                      self.pos, win)
        self.last_window = win
        pbb.advance_positions(self.pos)
        self.sim.append(k, v, (self.t0 + i).numpy())
        self.q_last = q
        self.step_i += 1
        return out

    def t_now(self) -> np.ndarray:
        """Positions of the tokens of the last step."""
        return (self.t0 + self.step_i - 1).numpy()

    def oracle_out(self, seqs=None) -> np.ndarray:
        """Oracle output of the last step for the given sequences (all by default)."""
        w = self.w
        seqs = np.arange(w.batch) if seqs is None else np.asarray(seqs)
        i = self.step_i - 1
        # window of B+1 rows ending at the current token: positions t-B .. t
        lo = i  # history row of position t - B
        sel = torch.as_tensor(seqs)
        hk = self.hk[:, :, lo:w.B + i + 1].index_select(0, sel)
        hv = self.hv[:, :, lo:w.B + i + 1].index_select(0, sel)
        t = self.t_now()[seqs]
        return _expected(self.q_last[seqs], hk, hv, t, w.B, self.last_window)

    def check_rings(self) -> None:
        assert np.array_equal(ring_bytes_np(self.k_ring), self.sim.k), "K ring differs from the oracle's"
        assert np.array_equal(ring_bytes_np(self.v_ring), self.sim.v), "V ring differs from the oracle's"


class DeviceRun:
    """Full-size run: inputs generated on the GPU (same recipe), rings prefilled
    on the GPU; the oracle checks a sample of sequences, whose history rows and
    step inputs are copied back to the host."""

    def __init__(self, w: inputs.Workload, sample, device="cuda", window=None):
        self.w = w
        self.window = window
        self.dev = torch.device(device)
        self.dtype = inputs.torch_dtype(w)
        self.sample = np.asarray(sample)
        self.t0 = inputs.start_positions(w)
        self.pos = self.t0.to(torch.int32).to(self.dev)
        self.k_ring = torch.empty((w.batch, w.Hkv, w.B, w.d), dtype=self.dtype, device=self.dev)
        self.v_ring = torch.empty_like(self.k_ring)
        wk, wv = inputs.history_window(w, self.t0, device=self.dev)
        pbb.ring_prefill(wk, wv, self.pos, self.k_ring, self.v_ring)
        idx = torch.as_tensor(self.sample, device=self.dev)
        # host history of the sampled sequences: window then one row per step
        self.hk = [wk.index_select(0, idx).cpu()]
        self.hv = [wv.index_select(0, idx).cpu()]
        del wk, wv
        torch.cuda.empty_cache()
        n = len(self.sample)
        self.sim = oracle.RingSim(n, w.Hkv, w.d, w.B, w.elem_bytes)
        self.sim.replay(self.hk[0], self.hv[0], (self.t0[self.sample] - w.B).numpy())
        self.step_i = 0
        self.q_last = None

    def step(self):
        w, i = self.w, self.step_i
        q, k, v = inputs.step_inputs(w, i, device=self.dev)
        out = _decode(q, k, v, self.k_ring, self.v_ring, self.pos, self.window)
        self.out = out  # every sequence's output of this step, on the device
        pbb.advance_positions(self.pos)
        idx = torch.as_tensor(self.sample, device=self.dev)
        ks, vs = k.index_select(0, idx).cpu(), v.index_select(0, idx).cpu()
        self.hk.append(ks.unsqueeze(2))
        self.hv.append(vs.unsqueeze(2))
        self.q_last = q.index_select(0, idx).cpu()
        self.sim.append(ks, vs, (self.t0[self.sample] + i).numpy())
        self.step_i += 1
        return out.index_select(0, idx).cpu()

    def oracle_out(self) -> np.ndarray:
        w, i = self.w, self.step_i - 1
        hk = torch.cat(self.hk, dim=2)[:, :, i:w.B + i + 1]
        hv = torch.cat(self.hv, dim=2)[:, :, i:w.B + i + 1]
        t = (self.t0[self.sample] + i).numpy()
        return _expected(self.q_last, hk, hv, t, w.B, self.window)

    def check_rings(self) -> None:
        idx = torch.as_tensor(self.sample, device=self.dev)
        assert np.array_equal(ring_bytes_np(self.k_ring.index_select(0, idx)), self.sim.k)
        assert np.array_equal(ring_bytes_np(self.v_ring.index_select(0, idx)), self.sim.v)
