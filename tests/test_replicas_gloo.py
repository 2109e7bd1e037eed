"""Multi-process (world size 2, gloo, CPU) check of the benchmark's replica
path: every rank times its own replica, the job time is the maximum over
ranks, and rank 0 reports the whole-job value (units of all replicas / max
time).  No GPU and no data-path collective are involved."""
import os
import socket

import torch
import torch.distributed as dist
import torch.multiprocessing as mp


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, times, out):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port),
                      RANK=str(rank), WORLD_SIZE=str(world), LOCAL_RANK=str(rank))
    import bench
    d, r, ws, lr = bench.dist_setup("gloo")
    assert (r, ws, lr) == (rank, world, rank)
    bench.barrier(d)
    t = bench.max_over_ranks(d, times[rank], torch.device("cpu"))
    out[rank] = t
    d.destroy_process_group()


def test_max_over_ranks_gloo():
    world = 2
    times = [3.5, 7.25]
    out = mp.get_context("spawn").Manager().dict()
    mp.spawn(_worker, args=(world, _free_port(), times, out), nprocs=world, join=True)
    assert out[0] == out[1] == max(times)


def test_single_process_has_no_collective():
    import bench
    os.environ.pop("WORLD_SIZE", None)
    d, r, ws, lr = bench.dist_setup("gloo")
    assert d is None and (r, ws, lr) == (0, 1, 0)
    assert bench.max_over_ranks(None, 4.0, torch.device("cpu")) == 4.0
    assert not dist.is_initialized()
