"""GPU parity of the whole-sequence PBB backward (pbb_backward) against the fp64
oracle's gradients.

Accuracy criteria are the paper's for its BF16 backward checks against an
exact-union reference (relative L2 error at most 0.02 and cosine similarity at
least 0.9998, per gradient tensor), applied here per (sequence, KV head) slice
of dq, dk and dv. The GPU runs on bf16 q, k, v, dO and its own bf16 forward
output O (D = dO . O), with the softmax weights and dS rounded to bf16 as mma
operands; the oracle differentiates the exact attention of the same bf16 inputs
in fp64.
"""
import numpy as np
import pytest
import torch

import oracle
import paper_2606_02680_gb300 as pbb
from paper_2606_02680_gb300 import inputs

pytestmark = pytest.mark.gpu

REL_L2 = 0.02
COSINE = 0.9998


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


def upstream(w, device="cpu", rows=None):
    """Seeded N(0,1) upstream gradient dO [batch, Hq, n, d] (bf16); rows restricts it to positions."""
    g = torch.Generator().manual_seed(w.seed + 1000)
    do = torch.randn((w.batch, w.Hq, w.n, w.d), generator=g).to(torch.bfloat16)
    if rows is not None:
        keep = torch.zeros(w.n, dtype=torch.bool)
        keep[rows] = True
        do = torch.where(keep.view(1, 1, -1, 1), do, torch.zeros((), dtype=torch.bfloat16))
    return do.to(device)


def compare(got, ref, what, per_head_axis=1):
    """Paper criteria per (sequence, head) slice; slices whose reference is all zero must be zero."""
    got = np.asarray(got, dtype=np.float64)
    assert np.all(np.isfinite(got)), f"{what}: non-finite"
    worst_rel, worst_cos = 0.0, 1.0
    for bi in range(ref.shape[0]):
        for hh in range(ref.shape[per_head_axis]):
            g, r = got[bi, hh].ravel(), ref[bi, hh].ravel()
            nr = np.linalg.norm(r)
            if nr == 0.0:
                assert np.abs(g).max() <= 1e-6, f"{what}[{bi},{hh}]: nonzero where the reference is zero"
                continue
            rel = np.linalg.norm(g - r) / nr
            cos = float(g @ r / (np.linalg.norm(g) * nr)) if np.linalg.norm(g) > 0 else 0.0
            worst_rel, worst_cos = max(worst_rel, rel), min(worst_cos, cos)
    assert worst_rel <= REL_L2 and worst_cos >= COSINE, f"{what}: rel-L2 {worst_rel:.2e}, cosine {worst_cos:.6f}"
    return worst_rel, worst_cos


def run_backward(w, dout_rows=None):
    dev = torch.device("cuda")
    q, k, v = inputs.sequence_inputs(w)
    do = upstream(w, rows=dout_rows)
    qd, kd, vd, dod = q.to(dev), k.to(dev), v.to(dev), do.to(dev)
    out, lse = pbb.forward(qd, kd, vd, w.B)
    dq, dk, dv = pbb.backward(qd, kd, vd, out, dod, lse, w.B)
    torch.cuda.synchronize()
    rq, rk, rv = oracle.backward(q, k, v, do, w.B)
    res = {name: compare(got.cpu().numpy(), ref, f"{w.name} {name}")
           for name, got, ref in (("dq", dq, rq), ("dk", dk, rk), ("dv", dv, rv))}
    return res, (dq, dk, dv), (rq, rk, rv)


@pytest.mark.parametrize("group", [1, 2, 4, 8])
@pytest.mark.parametrize("d", [64, 128])
def test_groups_and_dims(group, d):
    w = inputs.SequenceWorkload(f"bwd_g{group}_d{d}", batch=2, Hq=2 * group, Hkv=2, d=d, B=128, n=300,
                                seed=150 + group + d)
    run_backward(w)


@pytest.mark.parametrize("B", [2, 4, 16, 48, 96, 1024])
def test_block_sizes(B):
    n = 1500 if B == 1024 else 333
    w = inputs.SequenceWorkload(f"bwd_B{B}", batch=1, Hq=8, Hkv=2, d=128, B=B, n=n, seed=160 + B)
    run_backward(w)


@pytest.mark.parametrize("group", [2, 4])
def test_long_shape_head_dim_64(group):
    """d 64 with B = 1024: the one-CTA shape (128-row query tiles in the dK/dV pass, three
    Q/dO stages at this head size) over ragged tiles and both half-blocks."""
    w = inputs.SequenceWorkload(f"bwd_d64_B1024_g{group}", batch=1, Hq=2 * group, Hkv=2, d=64, B=1024, n=1500,
                                seed=165 + group)
    run_backward(w)


@pytest.mark.parametrize("n", [1, 7, 65])
def test_short_sequences(n):
    w = inputs.SequenceWorkload(f"bwd_n{n}", batch=2, Hq=4, Hkv=1, d=64, B=32, n=n, seed=170 + n)
    run_backward(w)


def test_bridge_gradients_reach_the_previous_block():
    """The paper's multi-block check: upstream gradient only on the bridge queries
    128..191 (B = 128, h = 64), which attend to the previous block's keys 64..127.
    Those keys get nonzero dk/dv equal to the oracle's; keys outside 64..191 get zero."""
    w = inputs.SequenceWorkload("bwd_bridge", batch=1, Hq=8, Hkv=2, d=64, B=128, n=1024, seed=180)
    res, (dq, dk, dv), (rq, rk, rv) = run_backward(w, dout_rows=np.arange(128, 192))
    dk, dv = dk.cpu().numpy(), dv.cpu().numpy()
    prev = slice(64, 128)
    assert np.linalg.norm(rk[:, :, prev]) > 0 and np.linalg.norm(rv[:, :, prev]) > 0
    for got, ref in ((dk, rk), (dv, rv)):
        rel = np.linalg.norm(got[:, :, prev] - ref[:, :, prev]) / np.linalg.norm(ref[:, :, prev])
        assert rel <= REL_L2
        assert np.abs(got[:, :, :64]).max() == 0.0 and np.abs(got[:, :, 192:]).max() == 0.0


def test_deterministic():
    w = inputs.SequenceWorkload("bwd_det", batch=2, Hq=16, Hkv=4, d=128, B=512, n=2000, seed=190)
    dev = torch.device("cuda")
    q, k, v = (x.to(dev) for x in inputs.sequence_inputs(w))
    do = upstream(w, dev)
    out, lse = pbb.forward(q, k, v, w.B)
    g1 = pbb.backward(q, k, v, out, do, lse, w.B)
    g2 = pbb.backward(q, k, v, out, do, lse, w.B)
    for a, b in zip(g1, g2):
        assert torch.equal(a, b)


@pytest.mark.parametrize("B,d", [(128, 64), (1024, 128)])  # the short and the long shape
def test_gradient_alignment(B, d):
    """Gradients 32-byte aligned take 32-byte stores, ones only 16-byte aligned 16-byte stores:
    both hold the same bits."""
    w = inputs.SequenceWorkload("bwd_align", batch=1, Hq=8, Hkv=2, d=d, B=B, n=1500, seed=195)
    dev = torch.device("cuda")
    q, k, v = (x.to(dev) for x in inputs.sequence_inputs(w))
    do = upstream(w, dev)
    out, lse = pbb.forward(q, k, v, w.B)
    g1 = pbb.backward(q, k, v, out, do, lse, w.B)
    bufs = []
    for g in g1:
        buf = torch.empty(g.numel() + 16, dtype=torch.float32, device=dev)
        base = (-buf.data_ptr() % 32) // 4 + 4  # 16 bytes past a 32-byte boundary
        t = buf[base:base + g.numel()].view(g.shape)
        assert t.data_ptr() % 32 == 16
        bufs.append(t)
    g2 = pbb.backward(q, k, v, out, do, lse, w.B, dq=bufs[0], dk=bufs[1], dv=bufs[2])
    for a, b in zip(g1, g2):
        assert a.data_ptr() % 32 == 0 and torch.equal(a, b)


@pytest.mark.parametrize("name", ["fwd_b16_n8192_B128"])
def test_full_size(name):
    """The benchmark's B = 128 workload at full size (batch 16, Hq 8, Hkv 2, d 64, n 8192), every gradient."""
    run_backward(inputs.FORWARD_WORKLOADS[name])


def test_large_block_long_sequence():
    """B = 1024 over 4096 positions, d 128: key tiles whose queries span two half-blocks of 512."""
    w = inputs.SequenceWorkload("bwd_B1024_n4096", batch=1, Hq=8, Hkv=2, d=128, B=1024, n=4096, seed=195)
    run_backward(w)
