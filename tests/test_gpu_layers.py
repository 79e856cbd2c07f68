"""GPU parity of the multi-layer decode step (pbb_decode_step_layers): L layers
with their own rings and inputs, one shared position per sequence, one launch.
Each layer's output is checked against the fp64 decode oracle over that layer's
history and every layer's rings byte for byte against the ring simulator."""
import numpy as np
import pytest
import torch

from pbb_testlib import check_close, ring_bytes_np

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


def run_layers(w, L, steps, chunk=0):
    pbb.set_chunk_keys(chunk)
    dev = torch.device("cuda")
    dt = inputs.torch_dtype(w)
    t0 = inputs.start_positions(w)                       # shared by the layers
    layers = [w.with_(seed=w.seed + 101 * (l + 1)) for l in range(L)]
    hist = [inputs.history_window(wl, t0) for wl in layers]
    k_ring = torch.zeros((L, w.batch, w.Hkv, w.B, w.d), dtype=dt, device=dev)
    v_ring = torch.zeros_like(k_ring)
    pos = t0.to(torch.int32).to(dev)
    sims = []
    for l in range(L):
        pbb.ring_prefill(hist[l][0].to(dev), hist[l][1].to(dev), pos, k_ring[l], v_ring[l])
        sim = oracle.RingSim(w.batch, w.Hkv, w.d, w.B, w.elem_bytes)
        sim.replay(hist[l][0], hist[l][1], (t0 - w.B).numpy())
        sims.append(sim)
    hk = [[h[0]] for h in hist]
    hv = [[h[1]] for h in hist]
    for i in range(steps):
        ins = [inputs.step_inputs(wl, i) for wl in layers]
        q = torch.stack([x[0] for x in ins]).to(dev)
        k = torch.stack([x[1] for x in ins]).to(dev)
        v = torch.stack([x[2] for x in ins]).to(dev)
        out = pbb.decode_step_layers(q, k, v, k_ring, v_ring, pos).cpu()
        pbb.advance_positions(pos)
        t = (t0 + i).numpy()
        for l in range(L):
            hk[l].append(ins[l][1].unsqueeze(2))
            hv[l].append(ins[l][2].unsqueeze(2))
            sims[l].append(ins[l][1], ins[l][2], t)
            kk = torch.cat(hk[l], dim=2)[:, :, i:w.B + i + 1]
            vv = torch.cat(hv[l], dim=2)[:, :, i:w.B + i + 1]
            ref = oracle.attend(ins[l][0], kk, vv, s0=t - w.B, t=t, b=w.B)
            check_close(out[l], ref, w.dtype, f"layer {l} step {i}")
    for l in range(L):
        assert np.array_equal(ring_bytes_np(k_ring[l]), sims[l].k)
        assert np.array_equal(ring_bytes_np(v_ring[l]), sims[l].v)
    assert pbb.get_device_status() == pbb.PBB_OK


@pytest.mark.parametrize("chunk", [0, 64])
def test_three_layers_ragged(chunk):
    w = inputs.Workload("layers3", batch=4, Hq=16, Hkv=4, d=128, B=256, dtype="bf16", steps=0,
                        t0_lo=0, t0_hi=3000, seed=300)
    run_layers(w, 3, 40, chunk)


def test_fifteen_layers_batch_one():
    """The paper's hybrid has 15 local layers: one token of batch 1 through all of them."""
    w = inputs.Workload("layers15", batch=1, Hq=8, Hkv=2, d=64, B=128, dtype="bf16", steps=0,
                        t0_lo=0, t0_hi=1000, seed=301)
    run_layers(w, 15, 20)


def test_group8_tensor_core_layers():
    w = inputs.Workload("layers_g8", batch=3, Hq=16, Hkv=2, d=128, B=128, dtype="bf16", steps=0,
                        t0_lo=0, t0_hi=2000, seed=302)
    assert pbb.plan_kernel(2 * w.batch, w.Hq, w.Hkv, w.d, w.B) == "tensor_cores"
    run_layers(w, 2, 30)


@pytest.mark.parametrize("kernel", ["cuda_cores", "tensor_cores"])
def test_group6_layers(kernel):
    """Two local layers of the paper's model shape (12 query heads on 2 KV heads, d 64), on
    both kernels (the library's choice is the tensor cores)."""
    w = inputs.Workload("layers_g6", batch=3, Hq=12, Hkv=2, d=64, B=128, dtype="bf16", steps=0,
                        t0_lo=0, t0_hi=2000, seed=304)
    prev = pbb.set_kernel(kernel)
    try:
        assert pbb.plan_kernel(2 * w.batch, w.Hq, w.Hkv, w.d, w.B) == kernel
        run_layers(w, 2, 30)
    finally:
        pbb.set_kernel(prev)


def test_fp32_layers():
    w = inputs.Workload("layers_f32", batch=2, Hq=8, Hkv=2, d=64, B=128, dtype="f32", steps=0,
                        t0_lo=0, t0_hi=600, seed=303)
    run_layers(w, 4, 30)


def test_too_many_layers_rejected():
    dev = torch.device("cuda")
    lib = pbb.lib()
    rc = lib.pbb_decode_step_layers(None, None, None, None, None, None, None, 0, 4, 8, 2, 64, 128, 0, None)
    assert rc == pbb.PBB_ERR_INVALID_ARG
    rc = lib.pbb_decode_step_layers(None, None, None, None, None, None, None, 300, 300, 8, 2, 64, 128, 0, None)
    assert rc == pbb.PBB_ERR_UNSUPPORTED
