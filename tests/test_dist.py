"""Multi-rank host logic of bench.py on CPU: world size 2, gloo, 127.0.0.1.

The decode step shards by sequence with no data-path collective; the ranks
share only the timing barrier and a max / sum over ranks. This covers that
host logic without a GPU.
"""
import os
import socket
import sys

import pytest
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, q):
    os.environ.update(RANK=str(rank), LOCAL_RANK=str(rank), WORLD_SIZE=str(world),
                      MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    sys.path.insert(0, ROOT)
    import bench

    try:
        dist, r, w, local = bench.dist_setup()
        assert (r, w, local) == (rank, world, rank)
        out = {
            "weak": bench.shard_batch(512, r, w, "weak"),
            "strong": bench.shard_batch(513, r, w, "strong"),
            "max": bench.max_over_ranks(dist, 1.5 + r),
            "sum": bench.sum_over_ranks(dist, 10.0 * (r + 1)),
        }
        dist.barrier()
        dist.destroy_process_group()
        q.put((rank, out))
    except Exception as e:  # noqa: BLE001 - report to the parent
        q.put((rank, repr(e)))


def test_two_ranks_shard_and_reduce():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_rank_main, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    results = dict(q.get(timeout=120) for _ in procs)
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    for r in range(2):
        assert isinstance(results[r], dict), results[r]
        assert results[r]["weak"] == 512          # weak scaling: every rank keeps the full batch
        assert results[r]["max"] == 2.5           # the slowest rank's time
        assert results[r]["sum"] == 30.0          # units of all ranks
    assert results[0]["strong"] + results[1]["strong"] == 513


def test_reference_arm_other_ranks_exit_without_work(monkeypatch):
    sys.path.insert(0, ROOT)
    import bench

    monkeypatch.setenv("RANK", "1")
    monkeypatch.setenv("WORLD_SIZE", "2")
    monkeypatch.setattr(sys, "argv", ["bench.py", "--impl", "reference", "--steps", "1", "--warmup", "0"])
    bench.main()  # returns at once on rank 1 (no oracle work, no output)
