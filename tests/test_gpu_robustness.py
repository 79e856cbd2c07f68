"""Bounds and resume checks of the decode step at full size, in host-side forms.

Guard bands: every tensor a step reads or writes is carved out of a larger
buffer whose margins hold a canary pattern. Ring margins hold bf16 NaNs, so a
read past a ring would poison an output (caught by the parity check against the
fp64 oracle); written tensors must leave their margins untouched.

Checkpoint/resume: the rings and positions are copied to the host mid-run,
restored into fresh device buffers, and the run continues from them; outputs
and rings must equal the uninterrupted run's bit for bit (the paper's cache
checks compare full cache contents over long sequential runs, Appendix F.2).
"""
import numpy as np
import pytest
import torch

from pbb_testlib import DeviceRun, check_close

import oracle
import paper_2606_02680_gb300 as pbb
from paper_2606_02680_gb300 import inputs

pytestmark = pytest.mark.gpu

MARGIN = 64 * 1024  # bytes on each side of a guarded tensor (a multiple of 16: alignment kept)


@pytest.fixture(scope="module", autouse=True)
def _gpu():
    if not torch.cuda.is_available():
        pytest.skip("needs a GPU")
    from paper_2606_02680_gb300 import build as nvbuild

    nvbuild.build()
    oracle.build()
    torch.cuda.set_device(0)
    prev = pbb.set_chunk_keys(0)
    yield
    pbb.set_chunk_keys(prev)
    assert pbb.get_device_status() == pbb.PBB_OK


class Guarded:
    """A tensor of `shape`/`dtype` inside a byte buffer with MARGIN canary bytes on each side."""

    def __init__(self, shape, dtype, dev, canary_word: int):
        esize = torch.empty((), dtype=dtype).element_size()
        n = int(np.prod(shape))
        self.buf = torch.empty(2 * MARGIN + n * esize, dtype=torch.uint8, device=dev)
        self.buf.view(torch.int16).fill_(canary_word - 65536 if canary_word >= 32768 else canary_word)
        self.canary = self._margins().clone()
        self.t = self.buf[MARGIN:MARGIN + n * esize].view(dtype).view(shape)
        assert self.t.data_ptr() % 16 == 0

    def _margins(self):
        return torch.cat([self.buf[:MARGIN], self.buf[-MARGIN:]])

    def intact(self) -> bool:
        return torch.equal(self._margins(), self.canary)


BF16_NAN = 0x7FC1   # a quiet NaN: any read of it into a score or an output poisons the result
CANARY = 0xA55A     # plain pattern for buffers nothing should read outside


@pytest.mark.parametrize("name", ["bf16_b64_B2048_ragged", "bf16_b256_B4096_outlier", "headline"])
def test_guard_bands_full_size(name):
    """Configs 3 and 4 and the timed shape (batch 512, B 4096) with the library's plan: 3 steps
    into guarded rings, inputs and output; margins unchanged, outputs of sampled sequences
    within tolerance of the oracle (a ring read past its end would have read NaN)."""
    w = inputs.sweep_workload(512, 4096, steps=3) if name == "headline" else \
        inputs.WORKLOADS[name].with_(steps=3)
    dev = torch.device("cuda", 0)
    dt = inputs.torch_dtype(w)
    t0 = inputs.start_positions(w)
    kr = Guarded((w.batch, w.Hkv, w.B, w.d), dt, dev, BF16_NAN)
    vr = Guarded((w.batch, w.Hkv, w.B, w.d), dt, dev, BF16_NAN)
    pos = Guarded((w.batch,), torch.int32, dev, CANARY)
    out = Guarded((w.batch, w.Hq, w.d), torch.float32, dev, CANARY)
    q = Guarded((w.batch, w.Hq, w.d), dt, dev, BF16_NAN)
    kn = Guarded((w.batch, w.Hkv, w.d), dt, dev, BF16_NAN)
    vn = Guarded((w.batch, w.Hkv, w.d), dt, dev, BF16_NAN)
    pos.t.copy_(t0.to(torch.int32))
    hk, hv = inputs.history_window(w, t0, device=dev)
    pbb.ring_prefill(hk, hv, pos.t, kr.t, vr.t)
    sample = sorted(set(np.linspace(0, w.batch - 1, 12).astype(int).tolist()))
    idx = torch.as_tensor(sample, device=dev)
    hist_k, hist_v = [hk.index_select(0, idx).cpu()], [hv.index_select(0, idx).cpu()]
    del hk, hv
    for i in range(w.steps):
        qs, ks, vs = inputs.step_inputs(w, i, device=dev)
        q.t.copy_(qs)
        kn.t.copy_(ks)
        vn.t.copy_(vs)
        pbb.decode_step(q.t, kn.t, vn.t, kr.t, vr.t, pos.t, out=out.t)
        pbb.advance_positions(pos.t)
        hist_k.append(ks.index_select(0, idx).cpu().unsqueeze(2))
        hist_v.append(vs.index_select(0, idx).cpu().unsqueeze(2))
        t = (t0[sample] + i).numpy()
        ref = oracle.attend(qs.index_select(0, idx).cpu(), torch.cat(hist_k, 2)[:, :, i:],
                            torch.cat(hist_v, 2)[:, :, i:], s0=t - w.B, t=t, b=w.B)
        check_close(out.t.index_select(0, idx).cpu(), ref, w.dtype, f"{name} step {i}")
    torch.cuda.synchronize()
    assert pbb.get_device_status() == pbb.PBB_OK
    for g, what in ((kr, "K ring"), (vr, "V ring"), (out, "out"), (pos, "pos"), (q, "q"), (kn, "k_new"),
                    (vn, "v_new")):
        assert g.intact(), f"{name}: a margin of {what} changed"


@pytest.mark.parametrize("name,kernel", [("bf16_b64_B2048_ragged", "auto"), ("bf16_b256_B4096_outlier", "auto"),
                                         ("bf16_b64_B2048_ragged", "cuda_cores")])
def test_checkpoint_resume_is_bitwise(name, kernel):
    """Run 12 steps; after step 5 snapshot the rings and positions to pinned host memory and
    restore them into fresh device buffers; steps 6..11 from the restored state must give
    bitwise the same outputs and rings as the uninterrupted run. The restored run's last step
    is also checked against the oracle on sampled sequences."""
    w = inputs.WORKLOADS[name].with_(steps=12)
    dev = torch.device("cuda", 0)
    prev = pbb.set_kernel(kernel)
    try:
        sample = [0, 17, w.batch // 2, w.batch - 1]
        run = DeviceRun(w, sample)
        cut = 6
        for _ in range(cut):
            run.step()
        torch.cuda.synchronize()
        snap = [x.cpu().pin_memory() for x in (run.k_ring, run.v_ring, run.pos)]
        kr2 = torch.empty_like(run.k_ring)
        vr2 = torch.empty_like(run.v_ring)
        pos2 = torch.empty_like(run.pos)
        for d_, h_ in zip((kr2, vr2, pos2), snap):
            d_.copy_(h_, non_blocking=True)
        del snap
        for i in range(cut, w.steps):
            q, k, v = inputs.step_inputs(w, i, device=dev)
            out_b = pbb.decode_step(q, k, v, kr2, vr2, pos2)
            pbb.advance_positions(pos2)
            out_a = run.step()  # the uninterrupted run (sampled outputs on the host)
            assert torch.equal(out_b, run.out), f"step {i}: outputs differ after the resume"
        check_close(out_a, run.oracle_out(), w.dtype, f"{name} after resume")
        torch.cuda.synchronize()
        assert torch.equal(kr2.view(torch.int16), run.k_ring.view(torch.int16))
        assert torch.equal(vr2.view(torch.int16), run.v_ring.view(torch.int16))
        assert torch.equal(pos2, run.pos)
        run.check_rings()
    finally:
        pbb.set_kernel(prev)
