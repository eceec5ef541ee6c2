"""The benchmark's multi-rank arithmetic and the data-parallel gradient
exchange on CPU with the gloo backend (world size 2): the job time is the
slowest rank's, the job throughput counts every rank's samples, and the
all-reduced half-batch gradients equal the full batch's."""
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


def _dp_worker(rank, world, port, out):
    import numpy as np
    import oracle
    from paper_2602_07400_gb300 import synth
    from paper_2602_07400_gb300.pipeline import allreduce_gradients
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        wl = synth.Workload("dp", 64, 48, 4, 40.0, (64, 128, 192), (40, 40), 4, 5.0)
        conn1, th1, conn2, th2 = synth.network(wl, 0)
        x, labels = synth.blob_batch(wl.batch, wl.d, wl.classes, wl.sigma, seed=5)
        half = wl.batch // world
        sl = slice(rank * half, (rank + 1) * half)   # this rank's shard of the batch
        r = oracle.train_step(x.numpy()[sl], labels.numpy()[sl], wl.thresholds, conn1, th1, conn2, th2,
                              wl.classes, wl.tau)
        grads = [torch.from_numpy(r["dth1"].copy()), torch.from_numpy(r["dth2"].copy())]
        allreduce_gradients(grads)
        out[rank] = [g.numpy() for g in grads]
    finally:
        dist.destroy_process_group()


def test_data_parallel_gradient_exchange_gloo():
    # two ranks, each with half the batch: after the exchange both hold the
    # gradient of the full batch's mean loss
    import numpy as np
    import oracle
    from paper_2602_07400_gb300 import synth
    world = 2
    port = _free_port()
    mgr = mp.get_context("spawn").Manager()
    out = mgr.dict()
    mp.start_processes(_dp_worker, args=(world, port, out), nprocs=world, join=True, start_method="spawn")
    wl = synth.Workload("dp", 64, 48, 4, 40.0, (64, 128, 192), (40, 40), 4, 5.0)
    conn1, th1, conn2, th2 = synth.network(wl, 0)
    x, labels = synth.blob_batch(wl.batch, wl.d, wl.classes, wl.sigma, seed=5)
    full = oracle.train_step(x.numpy(), labels.numpy(), wl.thresholds, conn1, th1, conn2, th2, wl.classes, wl.tau)
    for rank in range(world):
        np.testing.assert_allclose(out[rank][0], full["dth1"], rtol=1e-10, atol=1e-15)
        np.testing.assert_allclose(out[rank][1], full["dth2"], rtol=1e-10, atol=1e-15)
    np.testing.assert_array_equal(out[0][0], out[1][0])


def test_traffic_record_digest_ignores_comments(tmp_path):
    # a capture stays valid across comment edits of its kernel source and
    # turns null once the code changes
    import bench
    a = tmp_path / "a.cu"
    a.write_text("// note\nint f(int x) { return x + 1; } /* block\ncomment */\n")
    b = tmp_path / "b.cu"
    b.write_text("int f(int x)   { return x + 1; }  // another note\n")
    c = tmp_path / "c.cu"
    c.write_text("int f(int x) { return x + 2; }\n")
    assert bench.code_digest(str(a)) == bench.code_digest(str(b))
    assert bench.code_digest(str(a)) != bench.code_digest(str(c))


def test_algorithmic_work_of_the_roofline_calls():
    # the per-call work the roofline divides by, restated from the counts:
    # layer-2 backward with input-gradient terms, 4(2^k-1) + 2^k operations
    # per (node, sample) and X + per-class dY rows + terms + 2 tables + conn;
    # hard layer, 2^k - 1 mux operations per (node, 32-sample word) and the
    # packed input and output words + conn + tables
    import bench
    from paper_2602_07400_gb300 import synth
    wl = synth.WORKLOADS["mnist"]
    work = bench.call_work(wl, 1024)
    B, w, k, K, C = 1024, 8000, 6, 64, 10
    assert work["backward2"][1] == 316 * w * B
    assert work["backward2"][0] == 4 * (w * B + C * B + w * k * B + 2 * w * K + w * k)
    assert work["forward2"][1] == 132 * w * B
    hw = synth.WORKLOADS["hard_cifar10"]
    N = 1 << 22
    W = N // 32
    hwork = bench.call_work(hw, N)
    assert hwork["hard1"][1] == 63 * 64000 * W
    assert hwork["hard1"][0] == 4 * (21504 * W + 64000 * W + 64000 * 6) + 8 * 64000


def test_integer_pipe_ceiling_is_the_sum_of_both_pipes():
    import bench
    roof = {"achieved": 10.0}
    rates = {"imad": {"T_lane_ops_s": 12.0}, "lop3": {"T_lane_ops_s": 8.0}}
    got = bench.integer_pipe_fraction(roof, rates)
    assert got["peak"] == 20.0 and abs(got["frac"] - 0.5) < 1e-12
