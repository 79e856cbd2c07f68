"""GPU parity at the full benchmark sizes, in the launch configuration the
benchmark times (the library's own split plan), against the fp64 oracle.

The oracle is brute force over every position up to t, so at these sizes it
checks samples: chosen steps for every sequence, every step for a few
sequences, and the rings byte for byte (whole rings where the host copy is
affordable, sampled sequences otherwise).
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
    prev = pbb.set_chunk_keys(0)  # the benchmark's plan
    yield
    pbb.set_chunk_keys(prev)
    assert pbb.get_device_status() == pbb.PBB_OK




def test_bf16_b32_B1024_aligned_4096_steps():
    """batch 32, Hq 16, Hkv 4, d 128, B 1024, 4096 steps from t = 0 (every phase of 4
    blocks): one rotating sequence every step, all sequences at phases 0, 1, h-1, h,
    h+1, B-1 of every block, rings compared whole every 1024 steps."""
    w = inputs.WORKLOADS["bf16_b32_B1024"]
    h = w.B // 2
    run = SequentialRun(w)
    for i in range(w.steps):
        out = run.step()
        r = i % w.B
        if r in (0, 1, h - 1, h, h + 1, w.B - 1):
            check_close(out.cpu(), run.oracle_out(), w.dtype, f"step {i}")
        else:
            s = i % w.batch
            check_close(out[s:s + 1].cpu(), run.oracle_out([s]), w.dtype, f"step {i} seq {s}")
        if (i + 1) % 1024 == 0:
            run.check_rings()
    assert pbb.get_device_status() == pbb.PBB_OK


def test_bf16_b64_B2048_ragged_256_steps():
    """batch 64, Hq 32, Hkv 8, B 2048, t0 ~ U[0, 512K): rings prefilled (checked whole),
    every sequence at steps 0, 1, 127, 255, two sequences every step."""
    w = inputs.WORKLOADS["bf16_b64_B2048_ragged"]
    run = SequentialRun(w)
    run.check_rings()
    for i in range(w.steps):
        out = run.step()
        if i in (0, 1, 127, 255):
            for lo in range(0, w.batch, 16):
                seqs = np.arange(lo, lo + 16)
                check_close(out[lo:lo + 16].cpu(), run.oracle_out(seqs), w.dtype, f"step {i}")
        else:
            seqs = [i % w.batch, (7 * i + 3) % w.batch]
            check_close(out[seqs].cpu(), run.oracle_out(seqs), w.dtype, f"step {i}")
    run.check_rings()


def test_bf16_b256_B4096_outliers_128_steps():
    """batch 256, Hq 16, Hkv 2 (group 8), B 4096, 1 % of K/V entries x20, t0 ~ U[0, 64K):
    every sequence at steps 0, 64, 127, two sequences every step, rings whole at the end."""
    w = inputs.WORKLOADS["bf16_b256_B4096_outlier"]
    run = SequentialRun(w)
    for i in range(w.steps):
        out = run.step()
        if i in (0, 64, 127):
            for lo in range(0, w.batch, 32):
                seqs = np.arange(lo, lo + 32)
                check_close(out[lo:lo + 32].cpu(), run.oracle_out(seqs), w.dtype, f"step {i}")
        else:
            seqs = [i % w.batch, (11 * i + 5) % w.batch]
            check_close(out[seqs].cpu(), run.oracle_out(seqs), w.dtype, f"step {i}")
    run.check_rings()


@pytest.mark.parametrize("batch", inputs.SWEEP_BATCHES)
@pytest.mark.parametrize("B", inputs.SWEEP_BLOCKS)
def test_sweep_point(batch, B):
    """Throughput-sweep shapes (Hq 32, Hkv 8, d 128, t0 ~ U[B, 2^20)) at full size:
    8 sampled sequences (first, last and spread), 3 steps, their rings byte for byte."""
    w = inputs.sweep_workload(batch, B, steps=3)
    sample = sorted(set(np.linspace(0, batch - 1, 8).astype(int).tolist()))
    run = DeviceRun(w, sample)
    for i in range(w.steps):
        out = run.step()
        check_close(out, run.oracle_out(), w.dtype, f"b{batch} B{B} step {i}")
    run.check_rings()
    assert pbb.get_device_status() == pbb.PBB_OK


def _edge_start_positions(batch: int, B: int, seed: int) -> torch.Tensor:
    """Start positions at chosen phases r = t mod B: the first sequences cycle through
    r in {0, 1, h-2, h-1, h, h+1, B-2, B-1} (a two-step run then crosses the bridge/no-bridge
    edge at h-1 -> h and the block boundary at B-1 -> 0), the rest are uniform; every block
    index is at least 1, so the bridge exists (Eq. pbb)."""
    h = B // 2
    edges = [0, 1, h - 2, h - 1, h, h + 1, B - 2, B - 1]
    g = torch.Generator().manual_seed(seed)
    blk = torch.randint(1, (1 << 20) // B, (batch,), generator=g, dtype=torch.int64)
    r = torch.randint(0, B, (batch,), generator=g, dtype=torch.int64)
    n_edge = min(batch, 4 * len(edges))
    r[:n_edge] = torch.tensor([edges[i % len(edges)] for i in range(n_edge)], dtype=torch.int64)
    return blk * B + r


def test_headline_every_sequence_at_edge_phases():
    """The benchmark's timed shape (batch 512, Hq 32, Hkv 8, d 128, B 4096, bf16; the library's
    plan, which runs group 4 padded to 8 on the tensor-core kernel) checked on EVERY sequence
    on two consecutive steps, with 32 sequences placed on the phase edges of Eq. (pbb) at
    B = 4096, and every sequence's rings byte for byte at the end against the oracle's ring
    simulator."""
    w = inputs.sweep_workload(512, 4096, steps=2)
    assert pbb.plan_kernel(w.batch, w.Hq, w.Hkv, w.d, w.B, torch.bfloat16) == "tensor_cores"
    # whole supports, several rounds per CTA: the step takes them longest first
    assert pbb.plan_support_order(w.batch, w.Hq, w.Hkv, w.d, w.B)
    dev = torch.device("cuda", 0)
    t0 = _edge_start_positions(w.batch, w.B, seed=23)
    pos = t0.to(torch.int32).to(dev)
    hk_d, hv_d = inputs.history_window(w, t0, device=dev)  # positions t0-B .. t0-1
    k_ring = torch.empty((w.batch, w.Hkv, w.B, w.d), dtype=torch.bfloat16, device=dev)
    v_ring = torch.empty_like(k_ring)
    pbb.ring_prefill(hk_d, hv_d, pos, k_ring, v_ring)
    new_k, new_v = [], []
    chunk = 32
    for i in range(w.steps):
        q, k, v = inputs.step_inputs(w, i, device=dev)
        out = pbb.decode_step(q, k, v, k_ring, v_ring, pos).cpu()
        pbb.advance_positions(pos)
        new_k.append(k.cpu())
        new_v.append(v.cpu())
        t = (t0 + i).numpy()
        qc = q.cpu()
        for lo in range(0, w.batch, chunk):
            sl = slice(lo, lo + chunk)
            # window of B+1 rows ending at the current token: positions t-B .. t
            wk = torch.cat([hk_d[sl].cpu()] + [x[sl].unsqueeze(2) for x in new_k], dim=2)[:, :, i:]
            wv = torch.cat([hv_d[sl].cpu()] + [x[sl].unsqueeze(2) for x in new_v], dim=2)[:, :, i:]
            ref = oracle.attend(qc[sl], wk, wv, s0=t[sl] - w.B, t=t[sl], b=w.B)
            check_close(out[sl], ref, w.dtype, f"step {i} sequences {lo}..{lo + chunk - 1}")
    assert pbb.get_device_status() == pbb.PBB_OK
    from pbb_testlib import ring_bytes_np

    for lo in range(0, w.batch, chunk):
        sl = slice(lo, lo + chunk)
        sim = oracle.RingSim(chunk, w.Hkv, w.d, w.B, 2)
        sim.replay(hk_d[sl].cpu(), hv_d[sl].cpu(), (t0[sl] - w.B).numpy())
        for i in range(w.steps):
            sim.append(new_k[i][sl], new_v[i][sl], (t0[sl] + i).numpy())
        assert np.array_equal(ring_bytes_np(k_ring[sl]), sim.k), f"K rings {lo}..{lo + chunk - 1}"
        assert np.array_equal(ring_bytes_np(v_ring[sl]), sim.v), f"V rings {lo}..{lo + chunk - 1}"


def test_support_order_plan():
    """Longest-first order only where every support is one work item on the tensor-core kernel
    and each resident CTA gets several: not for chunked plans, small batches or the CUDA cores."""
    assert pbb.plan_support_order(512, 32, 8, 128, 4096)             # the timed shape
    assert pbb.plan_support_order(512, 32, 8, 128, 4096, window=4096)  # its window control
    assert not pbb.plan_support_order(64, 32, 8, 128, 4096)          # chunked supports
    assert not pbb.plan_support_order(8, 32, 8, 128, 4096)           # latency-bound
    assert not pbb.plan_support_order(512, 32, 8, 128, 4096, dtype=torch.float32)  # CUDA cores
    with pytest.raises(pbb.PbbError):
        pbb.plan_support_order(512, 32, 8, 128, 4096, window=4097)
