"""GPU parity of the CUDA decode step against the fp64 oracle at small sizes.

Every output of every step is compared with the oracle, and the rings byte for
byte with the oracle's ring simulator. Sizes span several tiles, several CTAs
per support (so the Eq. (lse) combine runs) and ragged tails.
"""
import numpy as np
import pytest
import torch

from pbb_testlib import SequentialRun, check_close, ring_bytes_np

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


@pytest.fixture
def kernel():
    """pbb.set_kernel for the test, restored afterwards."""
    prev = pbb.set_kernel("auto")
    yield pbb.set_kernel
    pbb.set_kernel(prev)


def run_and_check(w, chunk_keys, chunk=0, check_every=1, ring_every=None):
    chunk_keys(chunk)
    run = SequentialRun(w)
    worst = 0.0
    for i in range(w.steps):
        out = run.step()
        if i % check_every == 0 or i == w.steps - 1:
            worst = max(worst, check_close(out.cpu(), run.oracle_out(), w.dtype, f"step {i}"))
        if ring_every and (i % ring_every == 0):
            run.check_rings()
    run.check_rings()
    assert pbb.get_device_status() == pbb.PBB_OK
    return worst


def test_fp32_one_layer_1024_steps(chunk_keys):
    """fp32, batch 1, Hq 8, Hkv 2, d 64, B 128, t = 0..1023 (8 block boundaries), every step."""
    w = inputs.WORKLOADS["fp32_b1_B128"]
    run_and_check(w, chunk_keys, chunk=0, ring_every=128)


def test_fp32_one_layer_split(chunk_keys):
    """The same workload with the support split across CTAs (32 keys each)."""
    w = inputs.WORKLOADS["fp32_b1_B128"].with_(steps=400)
    run_and_check(w, chunk_keys, chunk=32, ring_every=100)


@pytest.mark.parametrize("group", [1, 2, 4, 6, 8])
@pytest.mark.parametrize("d", [64, 128])
@pytest.mark.parametrize("chunk", [0, 32])
def test_bf16_groups_and_dims(chunk_keys, group, d, chunk):
    """bf16, every supported GQA group and head size, B = 96 (not a power of two,
    tiles straddle the ring end; CUDA-core kernel for every group), 3 blocks from
    t = 0, batch 3."""
    w = inputs.Workload(f"g{group}_d{d}", batch=3, Hq=2 * group, Hkv=2, d=d, B=96, dtype="bf16",
                        steps=3 * 96 + 5, t0_lo=0, t0_hi=1, seed=100 + group + d)
    chunk_keys(chunk)
    assert pbb.plan_kernel(w.batch, w.Hq, w.Hkv, w.d, w.B) == "cuda_cores"
    run_and_check(w, chunk_keys, chunk=chunk, check_every=1)


@pytest.mark.parametrize("group,d,dtype", [(4, 128, "bf16"), (8, 128, "bf16"), (4, 64, "f32"),
                                           (2, 128, "f32"), (6, 64, "bf16"), (6, 128, "f32")])
def test_ragged_prefilled(chunk_keys, group, d, dtype):
    """Ragged start positions with rings loaded by pbb_ring_prefill; every step checked."""
    w = inputs.Workload("ragged", batch=5, Hq=2 * group, Hkv=2, d=d, B=256, dtype=dtype,
                        steps=300, t0_lo=0, t0_hi=5000, seed=7 + group)
    run_and_check(w, chunk_keys, chunk=0)
    run_and_check(w, chunk_keys, chunk=64)


@pytest.mark.parametrize("which", ["cuda_cores", "tensor_cores"])
def test_paper_model_shape_group6(chunk_keys, kernel, which):
    """The paper's models (Sec. 5): 12 query heads on 2 KV heads, head size 64, block 128.
    GQA group 6 runs on either kernel's 8 query columns with two zero query rows that are
    never written (the library picks the tensor cores, B being a multiple of 64): batch 1 from t = 0 across
    5 block boundaries, every step, then ragged prefilled positions with every support
    split into 32-key chunks."""
    w = inputs.Workload("paper_g6", batch=1, Hq=12, Hkv=2, d=64, B=128, dtype="bf16",
                        steps=5 * 128 + 3, t0_lo=0, t0_hi=1, seed=612)
    assert pbb.plan_kernel(w.batch, w.Hq, w.Hkv, w.d, w.B) == "tensor_cores"
    kernel(which)
    assert pbb.plan_kernel(w.batch, w.Hq, w.Hkv, w.d, w.B) == which
    run_and_check(w, chunk_keys, ring_every=128)
    w = w.with_(name="paper_g6_ragged", batch=5, steps=200, t0_hi=50000, seed=613)
    run_and_check(w, chunk_keys, chunk=32)


def test_prefill_is_bit_exact(chunk_keys):
    w = inputs.Workload("prefill", batch=6, Hq=8, Hkv=2, d=128, B=64, dtype="bf16", steps=1,
                        t0_lo=0, t0_hi=200, seed=9)
    run = SequentialRun(w)
    run.check_rings()


@pytest.mark.parametrize("group", [1, 8])
def test_smallest_block(chunk_keys, group):
    """B = 2 (h = 1): the bridge is one position."""
    w = inputs.Workload("b2", batch=2, Hq=group, Hkv=1, d=64, B=2, dtype="bf16", steps=20,
                        t0_lo=0, t0_hi=1, seed=3)
    run_and_check(w, chunk_keys)


def test_first_token_output_is_its_value():
    w = inputs.Workload("t0", batch=4, Hq=8, Hkv=2, d=128, B=128, dtype="bf16", steps=1,
                        t0_lo=0, t0_hi=1, seed=5)
    run = SequentialRun(w)
    out = run.step().cpu()
    _, _, v = inputs.step_inputs(w, 0)
    ref = v.float().repeat_interleave(4, dim=1)
    assert torch.equal(out, ref)


def test_deterministic_and_partition_invariant(chunk_keys):
    """Same inputs -> bitwise the same outputs and rings; with a fixed split, two
    half batches reproduce the full batch bit for bit."""
    chunk_keys(64)
    w = inputs.Workload("det", batch=8, Hq=16, Hkv=4, d=128, B=512, dtype="bf16", steps=1,
                        t0_lo=1000, t0_hi=100000, seed=21)
    dev = torch.device("cuda")
    t0 = inputs.start_positions(w)
    wk, wv = inputs.history_window(w, t0)
    q, k, v = inputs.step_inputs(w, 0)
    outs, rings = [], []
    for rep in range(2):
        pos = t0.to(torch.int32).to(dev)
        kr = torch.zeros((w.batch, w.Hkv, w.B, w.d), dtype=torch.bfloat16, device=dev)
        vr = torch.zeros_like(kr)
        pbb.ring_prefill(wk.to(dev), wv.to(dev), pos, kr, vr)
        outs.append(pbb.decode_step(q.to(dev), k.to(dev), v.to(dev), kr, vr, pos).cpu())
        rings.append((kr.cpu(), vr.cpu()))
    assert torch.equal(outs[0], outs[1])
    assert torch.equal(rings[0][0].view(torch.int16), rings[1][0].view(torch.int16))
    halves = []
    for sl in (slice(0, 4), slice(4, 8)):
        pos = t0[sl].to(torch.int32).to(dev)
        kr = torch.zeros((4, w.Hkv, w.B, w.d), dtype=torch.bfloat16, device=dev)
        vr = torch.zeros_like(kr)
        pbb.ring_prefill(wk[sl].contiguous().to(dev), wv[sl].contiguous().to(dev), pos, kr, vr)
        halves.append(pbb.decode_step(q[sl].contiguous().to(dev), k[sl].contiguous().to(dev),
                                      v[sl].contiguous().to(dev), kr, vr, pos).cpu())
    assert torch.equal(torch.cat(halves), outs[0])


def test_negative_position_flagged_and_others_correct():
    w = inputs.Workload("neg", batch=3, Hq=8, Hkv=2, d=128, B=64, dtype="bf16", steps=1,
                        t0_lo=0, t0_hi=1, seed=8)
    dev = torch.device("cuda")
    pos = torch.tensor([5, -1, 0], dtype=torch.int32, device=dev)
    kr = torch.zeros((3, 2, 64, 128), dtype=torch.bfloat16, device=dev)
    vr = torch.zeros_like(kr)
    q, k, v = inputs.step_inputs(w, 0)
    out = torch.full((3, 8, 128), 7.0, device=dev)
    pbb.decode_step(q.to(dev), k.to(dev), v.to(dev), kr, vr, pos, out)
    assert pbb.get_device_status() == pbb.PBB_ERR_DEVICE_POSITION
    assert pbb.get_device_status() == pbb.PBB_OK  # cleared
    o = out.cpu()
    assert torch.all(o[1] == 7.0)  # the flagged sequence is left untouched
    assert torch.equal(o[2], v[2].float().repeat_interleave(4, dim=0))


def test_wait_timeout_reports_and_recovers(chunk_keys):
    """A wait limit of 0 makes the first wait on a bulk copy give up: the step
    reports PBB_ERR_DEVICE_TIMEOUT, and after the status is read the next step
    (normal limit) is correct again (the split counters were reset)."""
    chunk_keys(64)
    w = inputs.Workload("timeout", batch=4, Hq=8, Hkv=2, d=128, B=1024, dtype="bf16", steps=2,
                        t0_lo=5000, t0_hi=100000, seed=13)
    run = SequentialRun(w)
    kr0, vr0, pos0 = run.k_ring.clone(), run.v_ring.clone(), run.pos.clone()
    try:
        pbb.set_wait_timeout_ns(0)
        q, k, v = inputs.step_inputs(w, 0)
        dev = run.dev
        pbb.decode_step(q.to(dev), k.to(dev), v.to(dev), run.k_ring, run.v_ring, run.pos)
        assert pbb.get_device_status() == pbb.PBB_ERR_DEVICE_TIMEOUT
    finally:
        pbb.set_wait_timeout_ns(1_000_000_000)
    run.k_ring.copy_(kr0)
    run.v_ring.copy_(vr0)
    run.pos.copy_(pos0)
    out = run.step()
    check_close(out.cpu(), run.oracle_out(), "bf16", "after timeout")
    assert pbb.get_device_status() == pbb.PBB_OK


def test_graph_capture_matches_eager(chunk_keys):
    """Steps captured in a CUDA graph (after reserve_workspace) match eager steps bit for bit."""
    w = inputs.Workload("graph", batch=4, Hq=16, Hkv=4, d=128, B=256, dtype="bf16", steps=1,
                        t0_lo=300, t0_hi=3000, seed=31)
    dev = torch.device("cuda")
    t0 = inputs.start_positions(w)
    wk, wv = inputs.history_window(w, t0)
    q, k, v = (x.to(dev) for x in inputs.step_inputs(w, 0))
    n = 10

    def fresh():
        pos = t0.to(torch.int32).to(dev)
        kr = torch.zeros((w.batch, w.Hkv, w.B, w.d), dtype=torch.bfloat16, device=dev)
        vr = torch.zeros_like(kr)
        pbb.ring_prefill(wk.to(dev), wv.to(dev), pos, kr, vr)
        return pos, kr, vr

    pos, kr, vr = fresh()
    out_e = torch.empty((w.batch, w.Hq, w.d), device=dev)
    for _ in range(n):
        pbb.decode_step(q, k, v, kr, vr, pos, out_e)
        pbb.advance_positions(pos)
    torch.cuda.synchronize()

    s = torch.cuda.Stream()
    pbb.reserve_workspace(w.batch, w.Hq, w.Hkv, w.d, w.B, stream=s)  # the capture stream's workspace
    pos2, kr2, vr2 = fresh()
    out_g = torch.empty_like(out_e)
    torch.cuda.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=s):
        pbb.decode_step(q, k, v, kr2, vr2, pos2, out_g)
        pbb.advance_positions(pos2)
    for _ in range(n):
        g.replay()
    torch.cuda.synchronize()
    assert torch.equal(out_g, out_e)
    assert torch.equal(kr2.view(torch.int16), kr.view(torch.int16))
    assert torch.equal(pos2, pos)


def test_host_resident_step_matches_device_step():
    w = inputs.Workload("host", batch=4, Hq=8, Hkv=2, d=128, B=128, dtype="bf16", steps=1,
                        t0_lo=0, t0_hi=1000, seed=41)
    dev = torch.device("cuda")
    t0 = inputs.start_positions(w)
    wk, wv = inputs.history_window(w, t0)
    q, k, v = inputs.step_inputs(w, 0)
    outs = []
    for host in (False, True):
        pos = t0.to(torch.int32).to(dev)
        kr = torch.zeros((w.batch, w.Hkv, w.B, w.d), dtype=torch.bfloat16, device=dev)
        vr = torch.zeros_like(kr)
        pbb.ring_prefill(wk.to(dev), wv.to(dev), pos, kr, vr)
        if host:
            st = pbb.HostStep(w.batch, w.Hq, w.Hkv, w.d, torch.bfloat16, dev)
            out_h = torch.empty((w.batch, w.Hq, w.d), dtype=torch.float32).pin_memory()
            pbb.decode_step_host(q.pin_memory(), k.pin_memory(), v.pin_memory(), kr, vr, pos, out_h, st)
            torch.cuda.synchronize()
            outs.append(out_h.clone())
        else:
            outs.append(pbb.decode_step(q.to(dev), k.to(dev), v.to(dev), kr, vr, pos).cpu())
    assert torch.equal(outs[0], outs[1])


def test_ring_alloc_zeroed_and_usable():
    rings = pbb.ring_alloc(2, 2, 128, 64, torch.bfloat16)
    try:
        torch.cuda.synchronize()
        assert rings.k.shape == (2, 2, 64, 128) and rings.k.dtype == torch.bfloat16
        assert int(rings.k.view(torch.int16).abs().sum()) == 0
        w = inputs.Workload("alloc", batch=2, Hq=8, Hkv=2, d=128, B=64, dtype="bf16", steps=1,
                            t0_lo=0, t0_hi=1, seed=2)
        q, k, v = (x.cuda() for x in inputs.step_inputs(w, 0))
        pos = torch.zeros(2, dtype=torch.int32, device="cuda")
        out = pbb.decode_step(q, k, v, rings.k, rings.v, pos)
        assert torch.equal(out.cpu(), v.cpu().float().repeat_interleave(4, dim=1))
        assert torch.equal(rings.k[:, :, 0].cpu().view(torch.int16), k.cpu().view(torch.int16))
    finally:
        rings.free()


def test_large_positions_near_int32_max(chunk_keys):
    """Positions up to 2^31 - 1: the block arithmetic stays exact."""
    w = inputs.Workload("bigt", batch=2, Hq=8, Hkv=2, d=128, B=1024, dtype="bf16", steps=40,
                        t0_lo=(1 << 31) - 1 - 45, t0_hi=(1 << 31) - 1 - 40, seed=51)
    # the oracle tests the predicate at every s <= t (about 2^31 per sequence): check two steps
    run_and_check(w, chunk_keys, chunk=0, check_every=w.steps)


def test_large_block(chunk_keys):
    """B = 2^16 at batch 1: supports of up to 65,535 ring keys split across many CTAs."""
    w = inputs.Workload("bigB", batch=1, Hq=4, Hkv=1, d=128, B=1 << 16, dtype="bf16", steps=3,
                        t0_lo=(1 << 16) * 3 + 100, t0_hi=(1 << 16) * 4, seed=61)
    run_and_check(w, chunk_keys, chunk=0)


@pytest.mark.parametrize("B", [64, 128, 256])
@pytest.mark.parametrize("d", [64, 128])
@pytest.mark.parametrize("chunk", [0, 64])
def test_bf16_group8_tensor_core_path(chunk_keys, B, d, chunk):
    """bf16 with GQA group 8 and B a multiple of 64 runs the tensor-core kernel
    (TMA-swizzled tiles, mma.sync for Q.K^T and P.V): every step of 3 blocks from
    t = 0 (first-block, bridge and partial tiles), batch 3, against the oracle."""
    w = inputs.Workload(f"tc_B{B}_d{d}", batch=3, Hq=16, Hkv=2, d=d, B=B, dtype="bf16",
                        steps=3 * B + 3, t0_lo=0, t0_hi=1, seed=300 + B + d)
    chunk_keys(chunk)
    assert pbb.plan_kernel(w.batch, w.Hq, w.Hkv, w.d, w.B) == "tensor_cores"
    run_and_check(w, chunk_keys, chunk=chunk)


@pytest.mark.parametrize("group", [4, 6])
@pytest.mark.parametrize("B", [64, 256])
@pytest.mark.parametrize("d", [64, 128])
@pytest.mark.parametrize("chunk", [0, 64])
def test_bf16_padded_group_tensor_core_path(chunk_keys, kernel, group, B, d, chunk):
    """GQA groups 4 and 6 on the tensor-core kernel: the score tile's 8 query columns hold the
    group's heads and zero rows for the rest, whose outputs are never written. Every step of
    3 blocks from t = 0, batch 3, against the oracle; the output rows of neighbouring KV
    groups must come out untouched by the padded heads."""
    w = inputs.Workload(f"tcpad_g{group}_B{B}_d{d}", batch=3, Hq=2 * group, Hkv=2, d=d, B=B,
                        dtype="bf16", steps=3 * B + 3, t0_lo=0, t0_hi=1, seed=400 + group + B + d)
    chunk_keys(chunk)
    kernel("tensor_cores")  # batch 3 alone would stay on the CUDA cores
    assert pbb.plan_kernel(w.batch, w.Hq, w.Hkv, w.d, w.B) == "tensor_cores"
    run_and_check(w, chunk_keys, chunk=chunk)


@pytest.mark.parametrize("group", [4, 6, 8])
@pytest.mark.parametrize("d", [64, 128])
def test_bf16_tensor_core_ragged_outliers(chunk_keys, kernel, group, d):
    """Tensor-core path with ragged prefilled rings and x20 outliers (large logits)."""
    kernel("tensor_cores")
    w = inputs.Workload("tc_outlier", batch=6, Hq=group, Hkv=1, d=d, B=512, dtype="bf16", steps=80,
                        t0_lo=0, t0_hi=20000, outlier_frac=0.01, outlier_scale=20.0, seed=77 + d + group)
    assert pbb.plan_kernel(w.batch, w.Hq, w.Hkv, w.d, w.B) == "tensor_cores"
    run_and_check(w, chunk_keys, chunk=0)
    run_and_check(w, chunk_keys, chunk=128)


def test_kernel_choice(kernel):
    """The library's choice: bf16 groups 4, 6 and 8 with B a multiple of 64 on the tensor cores,
    whatever the batch; fp32, groups 1 and 2 and blocks that are not a multiple of 64 on the
    CUDA cores. pbb_set_kernel overrides it within what each kernel supports."""
    import torch as _t
    assert pbb.plan_kernel(1, 16, 2, 128, 4096) == "tensor_cores"
    assert pbb.plan_kernel(512, 32, 8, 128, 4096) == "tensor_cores"
    assert pbb.plan_kernel(8, 32, 8, 128, 4096) == "tensor_cores"
    assert pbb.plan_kernel(32, 16, 4, 128, 1024) == "tensor_cores"
    assert pbb.plan_kernel(512, 12, 2, 64, 128) == "tensor_cores"  # the paper's heads, 1,024 supports
    assert pbb.plan_kernel(1, 12, 2, 64, 128) == "tensor_cores"
    assert pbb.plan_kernel(512, 16, 2, 128, 96) == "cuda_cores"
    assert pbb.plan_kernel(512, 32, 8, 128, 4096, _t.float32) == "cuda_cores"
    assert pbb.plan_kernel(512, 16, 8, 128, 4096) == "cuda_cores"  # group 2
    assert kernel("cuda_cores") == "auto"
    assert pbb.plan_kernel(512, 32, 8, 128, 4096) == "cuda_cores"
    assert pbb.plan_kernel(1, 16, 2, 128, 4096) == "cuda_cores"
    assert kernel("tensor_cores") == "cuda_cores"
    assert pbb.plan_kernel(1, 32, 8, 128, 4096) == "tensor_cores"
    assert pbb.plan_kernel(1, 16, 8, 128, 4096) == "cuda_cores"  # group 2: no tensor-core kernel
    with pytest.raises(ValueError):
        kernel("fastest")


def test_host_pipeline_matches_device_steps():
    """HostPipeline (host-resident inputs and outputs, copies overlapped across
    steps) gives bitwise the outputs and rings of plain device steps."""
    w = inputs.Workload("pipe", batch=4, Hq=16, Hkv=4, d=128, B=256, dtype="bf16", steps=6,
                        t0_lo=300, t0_hi=5000, seed=91)
    dev = torch.device("cuda")
    t0 = inputs.start_positions(w)
    wk, wv = inputs.history_window(w, t0)
    steps = [inputs.step_inputs(w, i) for i in range(w.steps)]
    results = []
    for mode in ("device", "pipeline"):
        pos = t0.to(torch.int32).to(dev)
        kr = torch.zeros((w.batch, w.Hkv, w.B, w.d), dtype=torch.bfloat16, device=dev)
        vr = torch.zeros_like(kr)
        pbb.ring_prefill(wk.to(dev), wv.to(dev), pos, kr, vr)
        outs = []
        if mode == "device":
            for q, k, v in steps:
                outs.append(pbb.decode_step(q.to(dev), k.to(dev), v.to(dev), kr, vr, pos).cpu())
                pbb.advance_positions(pos)
        else:
            pipe = pbb.HostPipeline(w.batch, w.Hq, w.Hkv, w.d, torch.bfloat16, dev)
            host_out = [torch.empty((w.batch, w.Hq, w.d)).pin_memory() for _ in steps]
            for (q, k, v), o in zip(steps, host_out):
                pipe.step(q.pin_memory(), k.pin_memory(), v.pin_memory(), kr, vr, pos, o)
            pipe.synchronize()
            outs = [o.clone() for o in host_out]
        torch.cuda.synchronize()
        results.append((outs, kr.cpu(), pos.cpu()))
    for a, b in zip(results[0][0], results[1][0]):
        assert torch.equal(a, b)
    assert torch.equal(results[0][1].view(torch.int16), results[1][1].view(torch.int16))
    assert torch.equal(results[0][2], results[1][2])
