"""The multi-GPU logic of bench.py on CPU: with world_size 2 over gloo, every
rank gets the slowest rank's time and the whole-job rate is the units of all
ranks over that time (independent replicas, no data-path collective)."""
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


def _rank_main(rank, world, port, out):
    os.environ.update({"MASTER_ADDR": "127.0.0.1", "MASTER_PORT": str(port), "RANK": str(rank),
                       "WORLD_SIZE": str(world), "LOCAL_RANK": str(rank)})
    sys.path.insert(0, ROOT)
    import torch.distributed as dist

    import bench

    r, w, local = bench.dist_setup("gloo")
    assert (r, w, local) == (rank, world, rank)
    seconds = 1.0 + rank  # rank 1 is the slow one
    slowest = bench.reduce_max(seconds, w, "cpu")
    rate, slow2 = bench.replica_throughput(1000.0, seconds, w, "cpu")
    bench.barrier(w)
    out[rank] = (slowest, rate, slow2)
    dist.destroy_process_group()


def test_replicas_take_the_slowest_rank():
    ctx = mp.get_context("spawn")
    manager = ctx.Manager()
    out = manager.dict()
    port = _free_port()
    procs = [ctx.Process(target=_rank_main, args=(r, 2, port, out)) for r in range(2)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(timeout=120)
    assert all(p.exitcode == 0 for p in procs)
    for r in range(2):
        slowest, rate, slow2 = out[r]
        assert slowest == pytest.approx(2.0) and slow2 == pytest.approx(2.0)
        assert rate == pytest.approx(2 * 1000.0 / 2.0)


def test_single_process_needs_no_group():
    sys.path.insert(0, ROOT)
    import bench

    assert bench.reduce_max(3.5, 1, "cpu") == 3.5
    assert bench.replica_throughput(10.0, 2.0, 1, "cpu") == (5.0, 2.0)
