"""The multi-GPU path of bench.py is replicas only: every rank runs the same
step on its own GPU, and rank 0 reports each timing's maximum over the ranks.
The reduction is checked here with two gloo ranks on the CPU."""
import os
import socket

import pytest

torch = pytest.importorskip("torch")
import torch.distributed as dist
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank(rank, world, port, out):
    import sys
    sys.path.insert(0, ROOT)
    import bench
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        dist.barrier()
        # each rank's own timings: rank r is slower on the first, faster on the second
        got = bench.max_over_ranks([10.0 + rank, 5.0 - rank], dist, "cpu")
        out[rank] = got
    finally:
        dist.destroy_process_group()


def test_replica_timings_reduce_to_the_slowest_rank():
    world = 2
    port = _free_port()
    with mp.Manager() as mgr:
        out = mgr.dict()
        mp.spawn(_rank, args=(world, port, out), nprocs=world, join=True)
        res = dict(out)
    assert res[0] == res[1] == [11.0, 5.0]


def test_single_process_keeps_its_values():
    import sys
    sys.path.insert(0, ROOT)
    import bench
    assert bench.max_over_ranks([3, 4.5], None, "cpu") == [3.0, 4.5]
