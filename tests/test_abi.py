"""CPU checks of the C ABI: the library loads, exports every symbol the header
declares, sizes rings as Appendix F.1 states, and rejects bad arguments before
touching the GPU. No compute call is made here."""
import ctypes
import json
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "pbb.h")


@pytest.fixture(scope="module")
def pbb():
    from paper_2606_02680_gb300 import build as nvbuild

    nvbuild.build()
    import paper_2606_02680_gb300 as pbb

    pbb.lib()
    return pbb


def declared_functions():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(pbb_[a-z0-9_]+)\s*\(", text)))


def test_header_declares_the_boundary():
    names = declared_functions()
    for must in ("pbb_ring_alloc", "pbb_decode_step", "pbb_decode_step_f32", "pbb_ring_prefill",
                 "pbb_get_device_status", "pbb_error_string"):
        assert must in names


def test_library_exports_every_declared_symbol(pbb):
    lib = ctypes.CDLL(pbb.lib_path)
    for name in declared_functions():
        assert hasattr(lib, name), name
    assert set(declared_functions()) == set(pbb.EXPORTS), "binding table out of sync with the header"


def test_ring_bytes_matches_appendix_f1(pbb):
    g = json.load(open(os.path.join(ROOT, "tests", "golden", "paper_counts.json")))["ring_bytes"]
    import torch

    one = pbb.ring_bytes(g["batch"], g["Hkv"], g["d"], g["b"], torch.bfloat16)
    assert 2 * one == g["bytes"]
    assert pbb.ring_bytes(2, 8, 128, 4096, torch.float32) == 2 * 8 * 128 * 4096 * 4
    assert pbb.ring_bytes(-1, 8, 128, 4096) == 0


def test_error_strings(pbb):
    for code in (0, -1, -2, -3, -4, -5, -6):
        assert pbb.error_string(code)
    assert "unknown" in pbb.error_string(-99)


@pytest.mark.parametrize(
    "batch,Hq,Hkv,d,B,code",
    [
        (1, 8, 2, 128, 127, -2),   # B odd
        (1, 8, 2, 128, 0, -1),     # B not positive
        (1, 8, 3, 128, 128, -2),   # Hq % Hkv != 0
        (1, 32, 2, 128, 128, -2),  # group 16 not supported
        (1, 8, 2, 96, 128, -2),    # d not supported
        (-1, 8, 2, 128, 128, -1),  # negative batch
        (1, 8, 2, 128, (1 << 20) + 2, -2),  # B too large
    ],
)
def test_bad_shapes_rejected_before_launch(pbb, batch, Hq, Hkv, d, B, code):
    lib = pbb.lib()
    rc = lib.pbb_decode_step(None, None, None, None, None, None, None, batch, Hq, Hkv, d, B, None)
    assert rc == code


def test_null_pointers_rejected(pbb):
    lib = pbb.lib()
    assert lib.pbb_decode_step(None, None, None, None, None, None, None, 2, 8, 2, 128, 128, None) == -1
    assert lib.pbb_ring_prefill(None, None, None, None, None, 2, 2, 128, 128, 0, None) == -1
    assert lib.pbb_advance_positions(None, 3, None) == -1


def test_misaligned_pointers_rejected(pbb):
    lib = pbb.lib()
    p = 0x1000  # never dereferenced: the alignment check fails first
    rc = lib.pbb_decode_step(p + 2, p, p, p, p, p, p, 2, 8, 2, 128, 128, None)
    assert rc == -1


def test_stream_read_arguments_checked_on_the_host(pbb):
    lib = pbb.lib()
    p = 0x10000  # never dereferenced: every check below fails, or returns, before any launch
    assert lib.pbb_stream_read(None, 1024, p, None) == -1
    assert lib.pbb_stream_read(p + 8, 1024, p, None) == -1       # buffer not 16-byte aligned
    assert lib.pbb_stream_read(p, 1000, p, None) == -1           # size not a multiple of 16
    assert lib.pbb_stream_read(p, 1024, p + 4, None) == -1       # sink not 8-byte aligned
    assert lib.pbb_stream_read(p, 1024, None, None) == -1
    assert lib.pbb_stream_read(None, 0, None, None) == 0         # nothing to read: no launch


def test_empty_batch_is_a_no_op(pbb):
    lib = pbb.lib()
    assert lib.pbb_decode_step(None, None, None, None, None, None, None, 0, 8, 2, 128, 128, None) == 0
    assert lib.pbb_ring_prefill(None, None, None, None, None, 0, 2, 128, 128, 0, None) == 0


def test_chunk_override_roundtrip(pbb):
    prev = pbb.set_chunk_keys(64)
    assert pbb.set_chunk_keys(prev) == 64
    with pytest.raises(pbb.PbbError):
        pbb.set_chunk_keys(-5)


def test_product_path_does_not_use_the_oracle():
    """The package never imports the oracle and has no CPU fallback."""
    pkg = os.path.join(ROOT, "paper_2606_02680_gb300")
    for dirpath, _, files in os.walk(pkg):
        for f in files:
            if f.endswith((".py", ".cu", ".h", ".cpp")):
                text = open(os.path.join(dirpath, f)).read()
                assert "import oracle" not in text and "from oracle" not in text, f
                assert "pbb_oracle" not in text, f


def test_group6_decode_only(pbb):
    """GQA group 6 (12 query heads on 2 KV heads) is a decode shape; the whole-sequence
    forward and backward, whose tiles stack the group's heads into 128 rows, refuse it
    before looking at any pointer. Batch 0 makes the decode calls no-ops."""
    lib = pbb.lib()
    assert lib.pbb_decode_step(None, None, None, None, None, None, None, 0, 12, 2, 64, 128, None) == 0
    assert lib.pbb_swa_decode_step(None, None, None, None, None, None, None, 0, 12, 2, 64, 128,
                                   128, 0, None) == 0
    assert lib.pbb_forward(None, None, None, None, None, 1, 12, 2, 128, 64, 128, 0, None) == -2
    assert lib.pbb_backward(None, None, None, None, None, None, None, None, None, None, 1, 12, 2,
                            128, 64, 128, None) == -2
    assert lib.pbb_decode_step(None, None, None, None, None, None, None, 0, 24, 2, 64, 128, None) == -2


def test_forward_plan_checks_before_the_device(pbb):
    import ctypes

    lib = pbb.lib()
    x = ctypes.c_int(0)
    assert lib.pbb_plan_forward(1, 8, 2, 64, 64, 128, None, ctypes.byref(x)) == -1
    assert lib.pbb_plan_forward(1, 12, 2, 64, 64, 128, ctypes.byref(x), ctypes.byref(x)) == -2  # group 6
    assert lib.pbb_plan_forward(1, 8, 2, 64, 96, 128, ctypes.byref(x), ctypes.byref(x)) == -2   # d 96


def test_kernel_choice_roundtrip(pbb):
    """pbb_set_kernel needs no device: it records the choice for later steps."""
    lib = pbb.lib()
    assert lib.pbb_set_kernel(5) == -1 and lib.pbb_set_kernel(-2) == -1
    prev = pbb.set_kernel("cuda_cores")
    try:
        assert pbb.set_kernel("tensor_cores") == "cuda_cores"
        assert pbb.set_kernel("auto") == "tensor_cores"
        with pytest.raises(ValueError):
            pbb.set_kernel("mma")
    finally:
        pbb.set_kernel(prev)


def test_window_checked_before_launch(pbb):
    """pbb_swa_decode_step: a window outside [1, B] is refused before anything
    else; batch 0 with a valid window is a no-op (no device work)."""
    lib = pbb.lib()
    for window, code in ((0, -1), (-1, -1), (129, -1), (1, 0), (128, 0)):
        rc = lib.pbb_swa_decode_step(None, None, None, None, None, None, None, 0, 8, 2, 128, 128,
                                     window, 0, None)
        assert rc == code, (window, rc)


def test_whole_sequence_arguments_checked_before_the_device(pbb):
    """pbb_forward, pbb_backward and pbb_ring_from_sequence refuse bad arguments (null or
    misaligned pointers, negative lengths, row counts past 32-bit TMA coordinates) and treat
    empty work as a no-op, all before any device call. Pointers are never dereferenced."""
    lib = pbb.lib()
    p = 0x1000
    # pbb_forward(q, k, v, out, lse, batch, Hq, Hkv, n, d, B, out_dtype, stream)
    fwd = lib.pbb_forward
    assert fwd(None, None, None, None, None, 0, 8, 2, 128, 64, 128, 0, None) == 0       # batch 0
    assert fwd(None, None, None, None, None, 1, 8, 2, 0, 64, 128, 0, None) == 0         # n 0
    assert fwd(None, None, None, None, None, 1, 8, 2, -1, 64, 128, 0, None) == -1       # n < 0
    assert fwd(p, p, p, p, None, 1, 8, 2, 128, 64, 128, 7, None) == -1                  # out dtype
    assert fwd(None, p, p, p, None, 1, 8, 2, 128, 64, 128, 0, None) == -1               # null q
    assert fwd(p, p, p, p + 8, None, 1, 8, 2, 128, 64, 128, 0, None) == -1              # out misaligned
    assert fwd(p, p, p, p, p + 2, 1, 8, 2, 128, 64, 128, 1, None) == -1                 # lse misaligned
    assert fwd(p, p, p, p, None, 1 << 12, 32, 8, 1 << 14, 128, 128, 0, None) == -2      # 2^31 rows
    assert fwd(p, p, p, p, None, 1, 8, 2, 128, 64, 127, 0, None) == -2                  # B odd
    # pbb_backward(q, k, v, out, dout, lse, delta, dq, dk, dv, batch, Hq, Hkv, n, d, B, stream)
    bwd = lib.pbb_backward
    nul = (None,) * 10
    assert bwd(*nul, 0, 8, 2, 128, 64, 128, None) == 0                                  # batch 0
    assert bwd(*nul, 1, 8, 2, 0, 64, 128, None) == 0                                    # n 0
    assert bwd(*nul, 1, 8, 2, -3, 64, 128, None) == -1                                  # n < 0
    ptrs = [p] * 10
    for i in range(10):                                                                 # each null pointer
        args = list(ptrs)
        args[i] = None
        assert bwd(*args, 1, 8, 2, 128, 64, 128, None) == -1, i
    for i, off in ((0, 8), (5, 2), (6, 2), (7, 4)):                                     # q, lse, delta, dq
        args = list(ptrs)
        args[i] = p + off
        assert bwd(*args, 1, 8, 2, 128, 64, 128, None) == -1, i
    assert bwd(*ptrs, 1 << 12, 32, 8, 1 << 14, 128, 128, None) == -2                    # 2^31 rows
    assert bwd(*ptrs, 1, 8, 2, 128, 80, 128, None) == -2                                # d 80
    # pbb_ring_from_sequence(k, v, n, k_ring, v_ring, batch, Hkv, d, B, dtype, stream)
    rfs = lib.pbb_ring_from_sequence
    assert rfs(None, None, 5, None, None, 0, 2, 64, 128, 0, None) == 0                  # batch 0
    assert rfs(None, None, -1, p, p, 1, 2, 64, 128, 0, None) == -1                      # n < 0
    assert rfs(None, None, 5, p, p, 1, 2, 64, 128, 0, None) == -1                       # null history
    assert rfs(p, p, 5, None, p, 1, 2, 64, 128, 0, None) == -1                          # null ring
    assert rfs(p + 4, p, 5, p, p, 1, 2, 64, 128, 0, None) == -1                         # misaligned


def test_binding_refuses_host_tensors(pbb):
    """No CPU fallback: every compute call of the binding raises on host tensors before the
    library runs anything."""
    import torch

    bf = torch.bfloat16
    batch, Hq, Hkv, d, B, n = 1, 8, 2, 64, 128, 16
    q = torch.zeros(batch, Hq, d, dtype=bf)
    kn = torch.zeros(batch, Hkv, d, dtype=bf)
    ring = torch.zeros(batch, Hkv, B, d, dtype=bf)
    pos = torch.zeros(batch, dtype=torch.int32)
    calls = [
        lambda: pbb.decode_step(q, kn, kn, ring, ring.clone(), pos),
        lambda: pbb.swa_decode_step(q, kn, kn, ring, ring.clone(), pos, window=B),
        lambda: pbb.decode_step_layers(q[None], kn[None], kn[None], ring[None], ring[None].clone(), pos),
        lambda: pbb.ring_prefill(ring, ring.clone(), pos, ring.clone(), ring.clone()),
        lambda: pbb.advance_positions(pos),
    ]
    qs = torch.zeros(batch, Hq, n, d, dtype=bf)
    ks = torch.zeros(batch, Hkv, n, d, dtype=bf)
    lse = torch.zeros(batch, Hq, n, dtype=torch.float32)
    calls += [
        lambda: pbb.forward(qs, ks, ks.clone(), B),
        lambda: pbb.backward(qs, ks, ks.clone(), qs.clone(), qs.clone(), lse, B),
        lambda: pbb.ring_from_sequence(ks, ks.clone(), ring.clone(), ring.clone()),
    ]
    for i, call in enumerate(calls):
        with pytest.raises(TypeError, match="CUDA tensor"):
            call()
