"""pbb_decode_step_noalloc through the C ABI: against pbb_decode_step and the fp64 oracle.

The no-allocation entry point is for callers that cannot allocate device memory
while they decode: a serving runtime that hands all of HBM to its own pool and
forbids any other allocation, or a loop that cannot afford the device-wide
synchronisation a cudaMalloc can bring. Its split scratch is a fixed array
inside the library instead of the workspace pbb_decode_step grows with
cudaMalloc. This file is collected last on purpose, so a run that stops at the
first failure has already run every other test; it also passes when run alone.
"""
import ctypes

import numpy as np
import pytest
import torch

from pbb_testlib import check_close, ring_bytes_np

import oracle

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def lib():
    if not torch.cuda.is_available():
        pytest.skip("needs a GPU")
    from paper_2606_02680_gb300 import build as nvbuild

    nvbuild.build()
    oracle.build()
    import paper_2606_02680_gb300 as pbb

    torch.cuda.set_device(0)
    prev = pbb.set_chunk_keys(0)  # the library's own split plan
    yield pbb
    pbb.set_chunk_keys(prev)


def _state(pbb, w, t0, wk, wv, dev):
    pos = t0.to(torch.int32).to(dev)
    kr = torch.zeros((w.batch, w.Hkv, w.B, w.d), dtype=torch.bfloat16, device=dev)
    vr = torch.zeros_like(kr)
    pbb.ring_prefill(wk, wv, pos, kr, vr)
    return pos, kr, vr


@pytest.mark.parametrize("Hq,Hkv,d,kernel", [(16, 4, 128, "auto"), (12, 2, 64, "auto"), (8, 4, 128, "auto"),
                                              (16, 4, 128, "cuda_cores"), (12, 2, 64, "cuda_cores")])
def test_noalloc_matches_decode_step_and_oracle_on_two_calls(lib, Hq, Hkv, d, kernel):
    pbb = lib
    from paper_2606_02680_gb300 import inputs

    prev_kernel = pbb.set_kernel(kernel)
    try:
        _noalloc_against_decode_step(pbb, inputs, Hq, Hkv, d)
    finally:
        pbb.set_kernel(prev_kernel)


def _noalloc_against_decode_step(pbb, inputs, Hq, Hkv, d):
    dev = torch.device("cuda", 0)
    # small batch: the plan splits every support across many CTAs, so the scratch is used;
    # (12, 2, 64) is the paper's model shape, GQA group 6; the library runs groups 4 and 6 on
    # the tensor cores and group 2 on the CUDA cores, and the cuda_cores cases force that kernel
    w = inputs.Workload("noalloc", batch=4, Hq=Hq, Hkv=Hkv, d=d, B=2048, dtype="bf16", steps=2,
                        t0_lo=2048, t0_hi=100000, seed=77 + Hq)
    assert pbb.plan_chunk_keys(w.batch, w.Hq, w.Hkv, w.d, w.B) < w.B - 1
    t0 = inputs.start_positions(w)
    wk, wv = inputs.history_window(w, t0, device=dev)
    pos_a, kr_a, vr_a = _state(pbb, w, t0, wk, wv, dev)
    pos_b, kr_b, vr_b = _state(pbb, w, t0, wk, wv, dev)
    # the oracle's side: host history (positions t0-B .. t0-1, then one row per step) and its
    # ring simulator
    hk, hv = [wk.cpu()], [wv.cpu()]
    sim = oracle.RingSim(w.batch, w.Hkv, w.d, w.B, 2)
    sim.replay(hk[0], hv[0], (t0 - w.B).numpy())
    stream = torch.cuda.current_stream()
    s = ctypes.c_void_p(stream.cuda_stream)
    L = pbb.lib()
    for step in range(2):
        q, k, v = inputs.step_inputs(w, step, device=dev)
        out_a = torch.empty((w.batch, w.Hq, w.d), dtype=torch.float32, device=dev)
        out_b = torch.full_like(out_a, float("nan"))
        rc = L.pbb_decode_step(q.data_ptr(), k.data_ptr(), v.data_ptr(), kr_a.data_ptr(),
                               vr_a.data_ptr(), pos_a.data_ptr(), out_a.data_ptr(), w.batch, w.Hq,
                               w.Hkv, w.d, w.B, s)
        assert rc == pbb.PBB_OK
        rc = L.pbb_decode_step_noalloc(q.data_ptr(), k.data_ptr(), v.data_ptr(), kr_b.data_ptr(),
                                       vr_b.data_ptr(), pos_b.data_ptr(), out_b.data_ptr(), w.batch,
                                       w.Hq, w.Hkv, w.d, w.B, s)
        assert rc == pbb.PBB_OK
        assert L.pbb_advance_positions(pos_a.data_ptr(), w.batch, s) == pbb.PBB_OK
        assert L.pbb_advance_positions(pos_b.data_ptr(), w.batch, s) == pbb.PBB_OK
        torch.cuda.synchronize()
        # same split plan and kernel, deterministic combine order: bitwise the same result
        assert torch.equal(out_a, out_b), step
        assert torch.equal(kr_a.view(torch.int16), kr_b.view(torch.int16))
        assert torch.equal(vr_a.view(torch.int16), vr_b.view(torch.int16))
        # and the fp64 oracle over the history window ending at the current token
        hk.append(k.cpu().unsqueeze(2))
        hv.append(v.cpu().unsqueeze(2))
        t = (t0 + step).numpy()
        sim.append(k.cpu(), v.cpu(), t)
        win_k = torch.cat(hk, dim=2)[:, :, step:w.B + step + 1]
        win_v = torch.cat(hv, dim=2)[:, :, step:w.B + step + 1]
        ref = oracle.attend(q.cpu(), win_k, win_v, s0=t - w.B, t=t, b=w.B)
        check_close(out_b.cpu(), ref, "bf16", f"no-alloc step {step}")
        assert np.array_equal(ring_bytes_np(kr_b), sim.k), "K ring differs from the oracle's"
        assert np.array_equal(ring_bytes_np(vr_b), sim.v), "V ring differs from the oracle's"
    assert L.pbb_get_device_status(s) == pbb.PBB_OK


def test_noalloc_rejects_steps_beyond_its_scratch(lib):
    """A step whose split partials exceed the fixed array is refused before any launch. The
    buffers are sized for the step all the same, so that a kernel launched by mistake would
    stay inside them instead of touching memory it does not own."""
    pbb = lib
    dev = torch.device("cuda", 0)
    batch, Hq, Hkv, d, B = 64, 32, 8, 128, 4096
    prev = pbb.set_chunk_keys(32)  # 128 CTAs per support: partials far beyond the fixed array
    try:
        q = torch.zeros((batch, Hq, d), dtype=torch.bfloat16, device=dev)
        kn = torch.zeros((batch, Hkv, d), dtype=torch.bfloat16, device=dev)
        vn = torch.zeros_like(kn)
        kr = torch.zeros((batch, Hkv, B, d), dtype=torch.bfloat16, device=dev)
        vr = torch.zeros_like(kr)
        pos = torch.full((batch,), 3 * B // 2, dtype=torch.int32, device=dev)
        out = torch.full((batch, Hq, d), -7.0, dtype=torch.float32, device=dev)
        rc = pbb.lib().pbb_decode_step_noalloc(q.data_ptr(), kn.data_ptr(), vn.data_ptr(), kr.data_ptr(),
                                               vr.data_ptr(), pos.data_ptr(), out.data_ptr(), batch, Hq,
                                               Hkv, d, B, None)
        assert rc == pbb.PBB_ERR_SCRATCH_LIMIT
        assert "scratch" in pbb.error_string(rc)
        torch.cuda.synchronize()
        assert bool((out == -7.0).all()), "a refused step must not write its output"
    finally:
        pbb.set_chunk_keys(prev)
