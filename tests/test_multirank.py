"""The benchmark's multi-GPU bookkeeping on two CPU ranks (gloo): ranks run
independent batches (no data exchange), the job time is the slowest rank's,
and the throughput counts every rank's images."""
import os
import socket

import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank(rank, world, port, out):
    import sys
    sys.path.insert(0, os.path.dirname(os.path.dirname(os.path.abspath(__file__))))
    import bench
    dist.init_process_group("gloo", init_method=f"tcp://127.0.0.1:{port}", rank=rank,
                            world_size=world)
    try:
        local_ms = 10.0 * (rank + 1)  # rank 1 is the slow one
        job_ms = bench.max_over_ranks(local_ms, torch.device("cpu"))
        out[rank] = (job_ms, bench.job_throughput(128, world, 5, job_ms / 1e3))
        dist.barrier()
    finally:
        dist.destroy_process_group()


def test_two_rank_timing_takes_the_slowest_rank():
    world, port = 2, _free_port()
    with mp.get_context("spawn").Manager() as m:  # (no fork of a threaded process)
        out = m.dict()
        mp.spawn(_rank, args=(world, port, out), nprocs=world, join=True)
        res = dict(out)
    assert res[0] == res[1]  # every rank sees the same job time
    job_ms, ips = res[0]
    assert job_ms == pytest.approx(20.0)
    assert ips == pytest.approx(128 * 2 * 5 / 0.020)
