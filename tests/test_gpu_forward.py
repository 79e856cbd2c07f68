"""GPU parity of the whole-sequence PBB forward (pbb_forward) against the fp64
oracle, and of the rings it leaves for decoding (pbb_ring_from_sequence).

Accuracy bound (derived from the kernel's arithmetic, written here). Scores
q.k accumulate exact bf16 products in fp32, and the exponentials are
2^-22-relative, so the output error comes from two roundings to bf16, whose
8-bit significand gives a unit roundoff of 2^-8:
  * the softmax weights are rounded to bf16 before P.V while the normaliser sums
    the unrounded weights, so |o - o_ref| <= 2^-8 max_s |v_s|;
  * a bf16 output adds |o| 2^-8.
A row passes when |o - o_ref| <= 2^-8 (max |v| of its sequence and head + |o_ref|) + 1e-5,
elementwise. The log-partition is a sum of unrounded fp32 weights: |lse - ref| <= 1e-4.
"""
import numpy as np
import pytest
import torch

import oracle
import paper_2606_02680_gb300 as pbb
from paper_2606_02680_gb300 import inputs
from pbb_testlib import ring_bytes_np

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


def check_rows(out, lse, ref_o, ref_lse, vmax, what=""):
    """out/ref_o [rows, d], lse/ref_lse [rows], vmax [rows] (max |v| of the row's KV head)."""
    out = np.asarray(out, dtype=np.float64)
    err = np.abs(out - ref_o)
    bound = 2.0 ** -8 * (vmax[:, None] + np.abs(ref_o)) + 1e-5
    assert np.all(np.isfinite(out)), f"{what}: non-finite output"
    worst = float((err / bound).max())
    assert worst <= 1.0, f"{what}: error {err.max():.3e} exceeds the bound (ratio {worst:.2f})"
    if lse is not None:
        le = np.abs(np.asarray(lse, dtype=np.float64) - ref_lse)
        assert le.max() <= 1e-4, f"{what}: lse error {le.max():.3e}"
    return float(err.max())


def run_full(w, out_dtype=torch.bfloat16, with_lse=True):
    """Forward on the GPU and the oracle on every row; returns the worst abs error."""
    q, k, v = inputs.sequence_inputs(w)
    dev = torch.device("cuda")
    out, lse = pbb.forward(q.to(dev), k.to(dev), v.to(dev), w.B, lse=with_lse, out_dtype=out_dtype)
    torch.cuda.synchronize()
    ref_o, ref_lse = oracle.forward(q, k, v, w.B)
    vmax = v.float().abs().amax(dim=(2, 3)).repeat_interleave(w.group, dim=1).numpy()  # [batch, Hq]
    n = w.n
    rows_vmax = np.repeat(vmax[:, :, None], n, axis=2).reshape(-1)
    return check_rows(out.float().cpu().numpy().reshape(-1, w.d), None if lse is None else lse.cpu().numpy().reshape(-1),
                      ref_o.reshape(-1, w.d), ref_lse.reshape(-1), rows_vmax, w.name)


@pytest.mark.parametrize("group", [1, 2, 4, 8])
@pytest.mark.parametrize("d", [64, 128])
def test_groups_and_dims(group, d):
    """Every group and head size, B = 128, n = 300 (several query tiles and a ragged
    tail), batch 2, Hkv 2: every output row and lse against the oracle."""
    w = inputs.SequenceWorkload(f"fwd_g{group}_d{d}", batch=2, Hq=2 * group, Hkv=2, d=d, B=128, n=300,
                                seed=50 + group + d)
    run_full(w)


@pytest.mark.parametrize("B", [2, 4, 16, 48, 64, 96, 1024])
def test_block_sizes(B):
    """Blocks smaller than a CTA's positions (h < QT: rows of one CTA start their
    supports at different half-blocks), not powers of two, and larger than a K/V tile."""
    n = 1500 if B == 1024 else 333
    w = inputs.SequenceWorkload(f"fwd_B{B}", batch=1, Hq=8, Hkv=2, d=128, B=B, n=n, seed=60 + B)
    run_full(w)


@pytest.mark.parametrize("group", [1, 2, 4, 8])
@pytest.mark.parametrize("d", [64, 128])
def test_long_blocks_groups_and_dims(group, d):
    """Long supports (B = 512, the 128-key-tile shape) for every group and head size;
    n = 777 gives an odd number of 128-row query tiles per (sequence, KV head) and a ragged
    last tile."""
    w = inputs.SequenceWorkload(f"fwd_long_g{group}_d{d}", batch=2, Hq=2 * group, Hkv=2, d=d, B=512,
                                n=777, seed=90 + group + d)
    run_full(w)


@pytest.mark.parametrize("d", [64, 128])
def test_paired_kernel_one_tile_items(d):
    """Many short sequences under a long block (n = 100, B = 512): every paired item has one
    K/V tile, so each CTA runs ten such items back to back, one extra iteration each. Its K and
    V producers then run furthest ahead of the issuing thread on the per-iteration barrier ring
    (2 x stages + 1 iterations: 9 at d = 64), which the ring must outlast."""
    w = inputs.SequenceWorkload(f"fwd_one_tile_d{d}", batch=384, Hq=8, Hkv=2, d=d, B=512, n=100,
                                seed=96 + d)
    assert pbb.plan_forward_query_tiles(w.batch, w.Hq, w.Hkv, w.n, w.d, w.B) == 2
    run_full(w)


@pytest.mark.parametrize("n", [1, 7, 8, 63, 64, 65])
def test_short_sequences(n):
    w = inputs.SequenceWorkload(f"fwd_n{n}", batch=3, Hq=4, Hkv=1, d=64, B=32, n=n, seed=70 + n)
    run_full(w)


def test_fp32_output_and_no_lse():
    w = inputs.SequenceWorkload("fwd_f32", batch=2, Hq=8, Hkv=2, d=128, B=256, n=700, seed=80)
    run_full(w, out_dtype=torch.float32)
    run_full(w, with_lse=False)


def test_outliers():
    """1 % of K/V entries x20: the bound scales with max |v|."""
    w = inputs.SequenceWorkload("fwd_outl", batch=2, Hq=16, Hkv=2, d=128, B=512, n=1200,
                                outlier_frac=0.01, outlier_scale=20.0, seed=81)
    run_full(w)


def test_first_position_is_its_value():
    """t = 0: the support is {0}, so out[:, j, 0] = v[:, j // G, 0] exactly (fp32 output)."""
    w = inputs.SequenceWorkload("fwd_t0", batch=2, Hq=8, Hkv=2, d=64, B=128, n=70, seed=82)
    q, k, v = (x.cuda() for x in inputs.sequence_inputs(w))
    out, _ = pbb.forward(q, k, v, w.B, out_dtype=torch.float32)
    assert torch.equal(out[:, :, 0], v[:, :, 0].float().repeat_interleave(4, dim=1))


def test_deterministic():
    w = inputs.SequenceWorkload("fwd_det", batch=2, Hq=16, Hkv=4, d=128, B=512, n=2000, seed=83)
    q, k, v = (x.cuda() for x in inputs.sequence_inputs(w))
    o1, l1 = pbb.forward(q, k, v, w.B)
    o2, l2 = pbb.forward(q, k, v, w.B)
    assert torch.equal(o1.view(torch.int16), o2.view(torch.int16)) and torch.equal(l1, l2)


@pytest.mark.parametrize("B,d", [(512, 128), (128, 64)])  # the paired and the one-item kernel
@pytest.mark.parametrize("out_dtype", [torch.bfloat16, torch.float32])
def test_output_alignment(B, d, out_dtype):
    """An output 32-byte aligned takes 32-byte stores, one only 16-byte aligned 16-byte stores:
    both hold the same bits."""
    w = inputs.SequenceWorkload("fwd_align", batch=2, Hq=8, Hkv=2, d=d, B=B, n=1100, seed=84)
    q, k, v = (x.cuda() for x in inputs.sequence_inputs(w))
    shape = (w.batch, w.Hq, w.n, w.d)
    numel = w.batch * w.Hq * w.n * w.d
    step = 16 // torch.tensor([], dtype=out_dtype).element_size()  # elements in 16 bytes
    buf = torch.empty(numel + 4 * step, dtype=out_dtype, device="cuda")
    base = (-buf.data_ptr() % 32) // buf.element_size()  # first 32-byte aligned element
    outs = []
    for off in (base, base + step):  # 32-byte aligned, then 16-byte only
        out = buf[off:off + numel].view(shape)
        assert out.data_ptr() % 32 == (0 if off == base else 16)
        outs.append(pbb.forward(q, k, v, w.B, out=out, out_dtype=out_dtype)[0].clone())
    bits = torch.int16 if out_dtype == torch.bfloat16 else torch.int32
    assert torch.equal(outs[0].view(bits), outs[1].view(bits))


def sampled_rows(w, count, rng):
    bi = rng.integers(0, w.batch, count)
    j = rng.integers(0, w.Hq, count)
    t = np.concatenate([rng.integers(0, w.n, count - 8), [0, 1, w.B // 2 - 1, w.B // 2, w.B, w.B + w.B // 2,
                                                          w.n - 2, w.n - 1]])
    return np.stack([bi, j, np.minimum(t, w.n - 1)], axis=1)


@pytest.mark.parametrize("name", list(inputs.FORWARD_WORKLOADS))
def test_full_size_sampled(name):
    """The benchmark's forward workloads at full size, in the launch the benchmark
    times: 256 sampled rows (random and phase edges) against the oracle, one
    (sequence, KV head) slice at a time."""
    w = inputs.FORWARD_WORKLOADS[name]
    dev = torch.device("cuda")
    q, k, v = inputs.sequence_inputs(w, device=dev)
    out, lse = pbb.forward(q, k, v, w.B)
    torch.cuda.synchronize()
    rows = sampled_rows(w, 256, np.random.default_rng(7))
    for bi in range(w.batch):
        for kvh in range(w.Hkv):
            sel = rows[(rows[:, 0] == bi) & (rows[:, 1] // w.group == kvh)]
            if len(sel) == 0:
                continue
            hs = slice(kvh * w.group, (kvh + 1) * w.group)
            qs = q[bi:bi + 1, hs].cpu()
            ks, vs = k[bi:bi + 1, kvh:kvh + 1].cpu(), v[bi:bi + 1, kvh:kvh + 1].cpu()
            local = np.stack([np.zeros(len(sel), dtype=np.int64), sel[:, 1] - kvh * w.group, sel[:, 2]], axis=1)
            ref_o, ref_l = oracle.forward(qs, ks, vs, w.B, rows=local)
            got = out[bi, sel[:, 1], sel[:, 2]].float().cpu().numpy()
            got_l = lse[bi, sel[:, 1], sel[:, 2]].cpu().numpy()
            vmax = np.full(len(sel), float(vs.float().abs().max()))
            check_rows(got, got_l, ref_o, ref_l, vmax, f"{name} seq {bi} kv {kvh}")
    assert pbb.get_device_status() == pbb.PBB_OK


@pytest.mark.parametrize("n,B", [(300, 128), (100, 128), (0, 64), (4096 + 37, 1024)])
def test_ring_from_sequence_then_decode(n, B):
    """Prefill n positions with the forward, load the rings from the sequence, then
    decode positions n .. n+20: rings bit-exact with the oracle's ring simulator
    (which replays the sequence), outputs against the decode oracle."""
    w = inputs.SequenceWorkload("fwd_ring", batch=2, Hq=8, Hkv=2, d=128, B=B, n=max(n, 1), seed=90 + n)
    dev = torch.device("cuda")
    q, k, v = inputs.sequence_inputs(w)
    k, v = k[:, :, :n].contiguous(), v[:, :, :n].contiguous()
    kr = torch.full((w.batch, w.Hkv, B, w.d), 3.0, dtype=torch.bfloat16, device=dev)  # stale bytes
    vr = kr.clone()
    pbb.ring_from_sequence(k.to(dev), v.to(dev), kr, vr)
    sim = oracle.RingSim(w.batch, w.Hkv, w.d, B, 2)
    if n > 0:
        sim.replay(k, v, np.zeros(w.batch, dtype=np.int64))
    assert np.array_equal(ring_bytes_np(kr), sim.k) and np.array_equal(ring_bytes_np(vr), sim.v)
    dw = inputs.Workload("dec", batch=w.batch, Hq=w.Hq, Hkv=w.Hkv, d=w.d, B=B, dtype="bf16", steps=20, seed=91)
    pos = torch.full((w.batch,), n, dtype=torch.int32, device=dev)
    hk, hv = [k], [v]
    for i in range(dw.steps):
        qs, ks, vs = inputs.step_inputs(dw, i)
        o = pbb.decode_step(qs.to(dev), ks.to(dev), vs.to(dev), kr, vr, pos)
        pbb.advance_positions(pos)
        hk.append(ks.unsqueeze(2))
        hv.append(vs.unsqueeze(2))
        t = n + i
        ref = oracle.attend(qs, torch.cat(hk, dim=2), torch.cat(hv, dim=2), s0=0, t=t, b=B)
        err = np.abs(o.cpu().numpy() - ref).max()
        assert err <= 1e-2, (t, err)
        sim.append(ks, vs, np.full(w.batch, t))
    assert np.array_equal(ring_bytes_np(kr), sim.k) and np.array_equal(ring_bytes_np(vr), sim.v)


def test_launch_shapes():
    """Long supports (B >= 512) run 128-key tiles with one CTA per SM (all 512 TMEM columns);
    short ones run 32-key tiles with three CTAs per SM at d = 64 (128 columns each) and
    64-key tiles with two at d = 128 (256 each): more CTAs overlap the per-item latencies
    of one- to four-tile items."""
    assert pbb.plan_forward(2, 32, 8, 32768, 128, 4096) == (128, 1)
    assert pbb.plan_forward(16, 8, 2, 8192, 64, 128) == (32, 3)
    assert pbb.plan_forward(16, 8, 2, 8192, 128, 128) == (64, 2)
    assert pbb.plan_forward(1, 8, 2, 0, 64, 128)[1] == 0  # no work
    # two query tiles per CTA where B is a multiple of 256 and the supports are long
    assert pbb.plan_forward_query_tiles(2, 32, 8, 32768, 128, 4096) == 2
    assert pbb.plan_forward_query_tiles(2, 32, 8, 4000, 64, 512) == 2
    assert pbb.plan_forward_query_tiles(1, 8, 2, 3000, 128, 640) == 1  # 640 / 2 not a multiple of 128
    assert pbb.plan_forward_query_tiles(16, 8, 2, 8192, 64, 128) == 1
    with pytest.raises(pbb.PbbError):
        pbb.plan_forward_query_tiles(1, 6, 4, 100, 64, 128)  # Hq not a multiple of Hkv

