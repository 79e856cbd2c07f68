"""GPU parity of the sliding-window control step (pbb_swa_decode_step) against
the fp64 oracle's window attention: support {t-w+1, ..., t} over the same
B-slot ring (Sec. 2.3; Sec. 3 on SWA with w = B in a B-slot ring).

Every output of every step is compared with the oracle and the rings byte for
byte with the oracle's ring simulator, which knows nothing of the pattern: the
ring contents depend only on the tokens appended.
"""
import numpy as np
import pytest
import torch

from pbb_testlib import DeviceRun, SequentialRun, check_close

import oracle
import paper_2606_02680_gb300 as pbb
from paper_2606_02680_gb300 import inputs

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _gpu():
    if not torch.cuda.is_available():
        pytest.skip("needs a GPU")
    from paper_2606_02680_gb300 import build as nvbuild

    nvbuild.build()
    oracle.build()
    torch.cuda.set_device(0)
    yield
    assert pbb.get_device_status() == pbb.PBB_OK


@pytest.fixture
def chunk_keys():
    prev = pbb.set_chunk_keys(0)
    yield pbb.set_chunk_keys
    pbb.set_chunk_keys(prev)


def run_and_check(w, window, check_every=1, ring_every=None):
    run = SequentialRun(w, window=window)
    for i in range(w.steps):
        out = run.step()
        if i % check_every == 0 or i == w.steps - 1:
            check_close(out.cpu(), run.oracle_out(), w.dtype, f"window {window} step {i}")
        if ring_every and i % ring_every == 0:
            run.check_rings()
    run.check_rings()
    assert pbb.get_device_status() == pbb.PBB_OK


@pytest.mark.parametrize("group", [1, 2, 4, 6, 8])
@pytest.mark.parametrize("d", [64, 128])
@pytest.mark.parametrize("chunk", [0, 32])
def test_window_B_groups_and_dims(chunk_keys, group, d, chunk):
    """w = B = 96 from t = 0: the warm-up (t < w-1) and then a window whose run of
    ring slots starts anywhere and wraps past slot B-1; batch 3, 3 blocks."""
    w = inputs.Workload(f"swa_g{group}_d{d}", batch=3, Hq=2 * group, Hkv=2, d=d, B=96,
                        dtype="bf16", steps=3 * 96 + 5, t0_lo=0, t0_hi=1, seed=200 + group + d)
    chunk_keys(chunk)
    run_and_check(w, window=w.B)


@pytest.mark.parametrize("window", [1, 2, 37, 64, 95])
def test_windows_shorter_than_the_ring(chunk_keys, window):
    """1 <= w < B over ragged prefilled rings (w = 1 attends to the current token alone)."""
    w = inputs.Workload("swa_w", batch=5, Hq=16, Hkv=4, d=128, B=96, dtype="bf16", steps=120,
                        t0_lo=0, t0_hi=3000, seed=300 + window)
    chunk_keys(0)
    run_and_check(w, window=window)
    chunk_keys(32)
    run_and_check(w, window=window, check_every=7)


@pytest.mark.parametrize("group,d,dtype", [(4, 128, "bf16"), (8, 128, "bf16"), (4, 64, "f32"),
                                           (1, 128, "f32")])
def test_window_B_ragged_prefilled(chunk_keys, group, d, dtype):
    w = inputs.Workload("swa_ragged", batch=5, Hq=2 * group, Hkv=2, d=d, B=256, dtype=dtype,
                        steps=300, t0_lo=0, t0_hi=5000, seed=17 + group)
    chunk_keys(0)
    run_and_check(w, window=w.B, check_every=3)
    chunk_keys(64)
    run_and_check(w, window=w.B, check_every=5)


def test_fp32_window_128_1024_steps(chunk_keys):
    """The fp32 batch-1 workload (Hq 8, Hkv 2, d 64, B 128), window 128, t = 0..1023."""
    chunk_keys(0)
    run_and_check(inputs.WORKLOADS["fp32_b1_B128"], window=128, ring_every=128)


def test_first_token_output_is_its_value():
    w = inputs.Workload("swa_t0", batch=4, Hq=8, Hkv=2, d=128, B=128, dtype="bf16", steps=1,
                        t0_lo=0, t0_hi=1, seed=5)
    run = SequentialRun(w, window=128)
    out = run.step().cpu()
    _, _, v = inputs.step_inputs(w, 0)
    assert torch.equal(out, v.float().repeat_interleave(4, dim=1))


def test_window_one_returns_the_current_value():
    """w = 1: the support is {t}, so o_j = v_t exactly for every head of the group."""
    w = inputs.Workload("swa_w1", batch=3, Hq=8, Hkv=2, d=64, B=64, dtype="bf16", steps=4,
                        t0_lo=100, t0_hi=5000, seed=6)
    run = SequentialRun(w, window=1)
    for i in range(w.steps):
        out = run.step().cpu()
        _, _, v = inputs.step_inputs(w, i)
        assert torch.equal(out, v.float().repeat_interleave(4, dim=1))


def test_switching_patterns_on_one_ring(chunk_keys):
    """PBB and window steps share the ring: alternating them step by step keeps
    the ring bit-exact and every output equal to its own pattern's oracle."""
    w = inputs.Workload("swa_mix", batch=4, Hq=16, Hkv=4, d=128, B=128, dtype="bf16", steps=300,
                        t0_lo=0, t0_hi=2000, seed=41)
    chunk_keys(0)
    run = SequentialRun(w)
    for i in range(w.steps):
        win = (None, 128, 64)[i % 3]
        out = run.step(window=win)
        check_close(out.cpu(), run.oracle_out(), w.dtype, f"step {i} window {win}")
    run.check_rings()


def test_window_B_positions_near_int32_max(chunk_keys):
    chunk_keys(0)
    w = inputs.Workload("swa_big_t", batch=3, Hq=8, Hkv=2, d=128, B=256, dtype="bf16", steps=40,
                        t0_lo=2**31 - 1000, t0_hi=2**31 - 60, seed=23)
    run_and_check(w, window=w.B)


def test_window_B_is_deterministic(chunk_keys):
    chunk_keys(64)
    w = inputs.Workload("swa_det", batch=8, Hq=16, Hkv=4, d=128, B=512, dtype="bf16", steps=1,
                        t0_lo=1000, t0_hi=100000, seed=22)
    dev = torch.device("cuda")
    t0 = inputs.start_positions(w)
    wk, wv = inputs.history_window(w, t0)
    q, k, v = (x.to(dev) for x in inputs.step_inputs(w, 0))
    outs = []
    for _ in range(2):
        pos = t0.to(torch.int32).to(dev)
        kr = torch.zeros((w.batch, w.Hkv, w.B, w.d), dtype=torch.bfloat16, device=dev)
        vr = torch.zeros_like(kr)
        pbb.ring_prefill(wk.to(dev), wv.to(dev), pos, kr, vr)
        outs.append(pbb.swa_decode_step(q, k, v, kr, vr, pos, window=w.B).cpu())
    assert torch.equal(outs[0], outs[1])


def test_bad_window_raises():
    dev = torch.device("cuda")
    kr = torch.zeros((1, 2, 64, 64), dtype=torch.bfloat16, device=dev)
    q = torch.zeros((1, 8, 64), dtype=torch.bfloat16, device=dev)
    kv = torch.zeros((1, 2, 64), dtype=torch.bfloat16, device=dev)
    pos = torch.zeros(1, dtype=torch.int32, device=dev)
    for bad in (0, 65, -3):
        with pytest.raises(pbb.PbbError) as e:
            pbb.swa_decode_step(q, kv, kv, kr, kr.clone(), pos, window=bad)
        assert e.value.code == pbb.PBB_ERR_INVALID_ARG


@pytest.mark.parametrize("batch,B", [(512, 4096), (64, 4096), (1, 1024)])
def test_full_size_window_B(batch, B):
    """Full throughput-sweep shapes (Hq 32, Hkv 8, d 128, t0 ~ U[B, 2^20)) with the
    library's own plan, window = B: 8 sampled sequences, 3 steps, their rings."""
    prev = pbb.set_chunk_keys(0)
    try:
        w = inputs.sweep_workload(batch, B, steps=3)
        sample = sorted(set(np.linspace(0, batch - 1, 8).astype(int).tolist()))
        run = DeviceRun(w, sample, window=B)
        for i in range(w.steps):
            out = run.step()
            check_close(out, run.oracle_out(), w.dtype, f"b{batch} B{B} step {i}")
        run.check_rings()
    finally:
        pbb.set_chunk_keys(prev)
    assert pbb.get_device_status() == pbb.PBB_OK


@pytest.fixture
def tensor_cores():
    prev = pbb.set_kernel("tensor_cores")
    yield
    pbb.set_kernel(prev)


@pytest.mark.parametrize("group,d", [(4, 128), (8, 128), (6, 64), (8, 64)])
@pytest.mark.parametrize("window", [1, 2, 33, 127, 128])
def test_windows_on_tensor_cores(chunk_keys, tensor_cores, group, d, window):
    """Window steps on the tensor-core kernel (B = 128, a multiple of two tiles). A window's
    run of ring slots starts at any slot and may wrap past slot B-1, while tiles start at slot
    multiples of 32: the first and last tiles of a run are masked outside it, and the slot
    being written (position t-B, outside the window) is never read. Ragged prefilled rings
    from positions near 0 (short runs in the first block) up to a few blocks; the library's
    plan, then 32-key chunks (every support split, so the epilogue warp's combine runs)."""
    w = inputs.Workload(f"swa_tc_g{group}_d{d}_w{window}", batch=3, Hq=2 * group, Hkv=2, d=d, B=128,
                        dtype="bf16", steps=40, t0_lo=0, t0_hi=700, seed=400 + 7 * group + d + window)
    chunk_keys(0)
    run_and_check(w, window=window)
    chunk_keys(32)
    run_and_check(w, window=window, check_every=3)


def test_window_on_both_kernels_against_the_oracle(chunk_keys):
    """The same window step on both kernels (which round P differently: fp32 weights on the
    CUDA cores, a bf16 high and low part on the tensor cores), each against the oracle."""
    chunk_keys(0)
    w = inputs.Workload("swa_tc_vs_cc", batch=6, Hq=32, Hkv=4, d=128, B=256, dtype="bf16", steps=1,
                        t0_lo=0, t0_hi=3000, seed=77)
    window = 200
    dev = torch.device("cuda")
    t0 = inputs.start_positions(w)
    wk, wv = inputs.history_window(w, t0)
    q, k, v = inputs.step_inputs(w, 0)
    t = t0.numpy()
    ref = oracle.attend_window(q, torch.cat([wk, k.unsqueeze(2)], 2), torch.cat([wv, v.unsqueeze(2)], 2),
                               s0=t - w.B, t=t, w=window)
    for kernel in ("tensor_cores", "cuda_cores"):
        prev = pbb.set_kernel(kernel)
        try:
            pos = t0.to(torch.int32).to(dev)
            kr = torch.zeros((w.batch, w.Hkv, w.B, w.d), dtype=torch.bfloat16, device=dev)
            vr = torch.zeros_like(kr)
            pbb.ring_prefill(wk.to(dev), wv.to(dev), pos, kr, vr)
            out = pbb.swa_decode_step(q.to(dev), k.to(dev), v.to(dev), kr, vr, pos, window=window).cpu()
        finally:
            pbb.set_kernel(prev)
        check_close(out, ref, "bf16", kernel)
