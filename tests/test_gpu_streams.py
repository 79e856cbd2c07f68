"""Decode steps of two independent batches issued on two CUDA streams without any ordering
between the streams (from one host thread, and from two), each checked against the fp64
oracle. Every stream gets its own library workspace (work queue, split counters, partials), so
steps that overlap on the GPU do not share scratch."""
import threading

import numpy as np
import pytest
import torch

from pbb_testlib import SequentialRun, check_close

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
    prev = pbb.set_chunk_keys(0)
    yield
    pbb.set_chunk_keys(prev)
    assert pbb.get_device_status() == pbb.PBB_OK


def _oracle_at(run: SequentialRun, i: int) -> np.ndarray:
    """Oracle output of step i of a run (every sequence), from the run's host history."""
    w = run.w
    q = inputs.step_inputs(w, i)[0]
    t = (run.t0 + i).numpy()
    return oracle.attend(q, run.hk[:, :, i:w.B + i + 1], run.hv[:, :, i:w.B + i + 1], s0=t - w.B, t=t, b=w.B)


# small batches: the library splits every support across CTAs, so each step uses the split
# counters and partials of its workspace; one runs on the tensor cores (group 8), one on the
# CUDA cores (group 2)
SHAPES = [inputs.Workload("stream_a", batch=4, Hq=16, Hkv=2, d=128, B=2048, dtype="bf16", steps=16,
                          t0_lo=2048, t0_hi=200000, seed=61),
          inputs.Workload("stream_b", batch=3, Hq=8, Hkv=4, d=64, B=1024, dtype="bf16", steps=16,
                          t0_lo=0, t0_hi=100000, seed=62)]


def _run_pair(threads: bool):
    dev = torch.device("cuda", 0)
    streams = [torch.cuda.Stream(device=dev) for _ in SHAPES]
    runs = []
    for w, s in zip(SHAPES, streams):
        with torch.cuda.stream(s):
            runs.append(SequentialRun(w))
    torch.cuda.synchronize()
    outs = [[None] * w.steps for w in SHAPES]

    def drive(j):
        with torch.cuda.stream(streams[j]):
            for i in range(SHAPES[j].steps):
                outs[j][i] = runs[j].step()

    if threads:
        ts = [threading.Thread(target=drive, args=(j,)) for j in range(len(SHAPES))]
        for t in ts:
            t.start()
        for t in ts:
            t.join()
    else:
        for i in range(max(w.steps for w in SHAPES)):  # interleaved issue, no cross-stream order
            for j in range(len(SHAPES)):
                if i < SHAPES[j].steps:
                    with torch.cuda.stream(streams[j]):
                        outs[j][i] = runs[j].step()
    torch.cuda.synchronize()
    assert pbb.get_device_status() == pbb.PBB_OK
    for j, run in enumerate(runs):
        for i in range(SHAPES[j].steps):
            check_close(outs[j][i].cpu(), _oracle_at(run, i), "bf16", f"stream {j} step {i}")
        run.check_rings()


def test_two_streams_interleaved_from_one_thread():
    assert pbb.plan_kernel(4, 16, 2, 128, 2048) == "tensor_cores"
    _run_pair(threads=False)


def test_two_streams_from_two_host_threads():
    _run_pair(threads=True)
