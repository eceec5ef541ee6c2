"""The benchmark's multi-rank arithmetic on CPU with the gloo backend
(world size 2): the job time is the slowest rank's, the job throughput
counts every rank's samples."""
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


def _worker(rank, world, port, out):
    import bench
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        # rank 1 is the slow one for the first value, rank 0 for the second
        got = bench.max_over_ranks([10.0 + 5.0 * rank, 7.0 - rank], "cpu")
        out[rank] = (got, bench.job_rate(world, 1024, 20, got[0]))
    finally:
        dist.destroy_process_group()


def test_max_over_ranks_and_job_rate_gloo():
    world = 2
    port = _free_port()
    mgr = mp.get_context("spawn").Manager()
    out = mgr.dict()
    mp.start_processes(_worker, args=(world, port, out), nprocs=world, join=True,
                       start_method="spawn")
    for r in range(world):
        got, rate = out[r]
        assert got == [15.0, 7.0]
        assert rate == pytest.approx(2 * 1024 * 20 / 15e-3)


def test_single_process_is_identity():
    import bench
    assert bench.max_over_ranks([3.0, 4.0], "cpu") == [3.0, 4.0]
    assert bench.job_rate(1, 1024, 10, 5.0) == pytest.approx(1024 * 10 / 5e-3)
