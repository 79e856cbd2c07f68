"""The read-roof probe pbb_stream_read (a measurement utility of the library): it returns without
error on buffers of whole 16 KiB chunks and with a ragged tail, sets no timeout bit, and folds the
tail's words into the sink; it checks its arguments on the host."""
import numpy as np
import pytest
import torch

import paper_2606_02680_gb300 as pbb

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _gpu():
    if not torch.cuda.is_available():
        pytest.skip("needs a GPU")
    from paper_2606_02680_gb300 import build as nvbuild

    nvbuild.build()
    torch.cuda.set_device(0)


@pytest.mark.parametrize("nbytes", [16384, 16384 * 1000, 16384 * 977 + 4096, 48, 64 << 20])
def test_stream_read_tail_checksum_and_no_timeout(nbytes):
    dev = torch.device("cuda", 0)
    g = torch.Generator().manual_seed(nbytes % 1000)
    host = torch.randint(0, 256, (nbytes,), generator=g, dtype=torch.uint8)
    buf = host.to(dev)
    sink = torch.zeros(1, dtype=torch.int64, device=dev)
    pbb.stream_read(buf, sink)
    torch.cuda.synchronize()
    got = int(sink.item())
    assert got >= 0, "a bounded wait on a bulk copy ran out"
    tail = host.numpy()[(nbytes // 16384) * 16384:].view(np.uint32)
    expect = int(np.bitwise_xor.reduce(tail)) if tail.size else 0
    assert got == expect


def test_stream_read_rejects_bad_arguments():
    dev = torch.device("cuda", 0)
    buf = torch.zeros(1024, dtype=torch.uint8, device=dev)
    sink = torch.zeros(1, dtype=torch.int64, device=dev)
    L = pbb.lib()
    assert L.pbb_stream_read(buf.data_ptr() + 8, 1008, sink.data_ptr(), None) == pbb.PBB_ERR_INVALID_ARG
    assert L.pbb_stream_read(buf.data_ptr(), 1000, sink.data_ptr(), None) == pbb.PBB_ERR_INVALID_ARG
    assert L.pbb_stream_read(buf.data_ptr(), 1024, sink.data_ptr() + 4, None) == pbb.PBB_ERR_INVALID_ARG
    assert L.pbb_stream_read(None, 1024, sink.data_ptr(), None) == pbb.PBB_ERR_INVALID_ARG
    assert L.pbb_stream_read(buf.data_ptr(), 0, sink.data_ptr(), None) == pbb.PBB_OK
