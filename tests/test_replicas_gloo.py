"""The bench's multi-GPU path is replicas only (the active-block step is a sequential chain of
Adam steps on one block): each rank runs the whole stage, the job's time is the slowest
rank's, and the value counts every rank's steps.  That host logic, checked with two gloo
processes on the CPU (127.0.0.1 rendezvous)."""
import os
import socket

import pytest

torch = pytest.importorskip("torch")
import torch.distributed as dist
import torch.multiprocessing as mp


def _free_port():
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    port = s.getsockname()[1]
    s.close()
    return port


def _worker(rank, world, port, times, out):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world), LOCAL_RANK=str(rank))
    import bench
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        r, w, local = bench.dist_env()
        assert (r, w, local) == (rank, world, rank)
        ms = bench.max_over_ranks(times[rank], w)
        out[rank] = (ms, bench.replica_value(3, 500, w, ms))
        # the oracle arm: ranks other than 0 return at once, without work
        if rank != 0:
            args = bench.parse(["--impl", "reference"])
            assert bench.run_reference(args) is None
        dist.barrier()
    finally:
        dist.destroy_process_group()


def test_two_replicas_report_the_slowest_rank_and_all_steps():
    world = 2
    times = [120.0, 180.0]
    mgr = mp.get_context("spawn").Manager()
    out = mgr.dict()
    mp.start_processes(_worker, args=(world, _free_port(), times, out), nprocs=world,
                       start_method="spawn", join=True)
    for r in range(world):
        ms, value = out[r]
        assert ms == 180.0
        assert value == pytest.approx(3 * 500 * 2 / 0.18)
