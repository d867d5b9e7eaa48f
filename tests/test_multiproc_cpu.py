"""The replica mode of bench.py (one process per GPU, no collective on the data
path: heads are independent) with world size 2 on the gloo backend, on CPU:
the barrier, the max over ranks of the step time, and the whole-job value."""
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


def _rank_main(rank, world, port, results):
    sys.path.insert(0, ROOT)
    os.environ.update({"RANK": str(rank), "LOCAL_RANK": str(rank), "WORLD_SIZE": str(world),
                       "MASTER_ADDR": "127.0.0.1", "MASTER_PORT": str(port)})
    import torch.distributed as dist

    import bench
    r, w, _ = bench.dist_setup(world, backend="gloo")
    assert (r, w) == (rank, world)
    bench.barrier(w)
    ms = 1.0 + rank  # rank 1 is the slower one
    results[rank] = (bench.max_over_ranks(ms, w), bench.weak_scaling_value(1000, w, bench.max_over_ranks(ms, w)))
    bench.barrier(w)
    dist.destroy_process_group()


def test_replica_mode_two_ranks_gloo():
    world = 2
    port = _free_port()
    with mp.Manager() as m:
        results = m.dict()
        mp.spawn(_rank_main, args=(world, port, results), nprocs=world, join=True)
        res = dict(results)
    assert res[0] == res[1] == (2.0, 1000 * 2 / 2e-3)
