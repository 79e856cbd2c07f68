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
