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
    # algorithmic bytes leave out the per-edge terms (implementation
    # overhead); the bytes moved carry them (written here, read by csr2)
    assert work["backward2"][0] == 4 * (w * B + C * B + 2 * w * K + w * k)
    assert work["backward2"][2] == work["backward2"][0] + 4 * w * k * B
    # the layer-2 backward with input gradient (backward2 + csr2) moves
    # X, the per-class dY rows, dX, the table and its gradient, the
    # connectivity and the CSR map once each
    w_in1 = 8000
    assert work["backward2"][0] + work["csr2"][0] == 4 * (w * B + C * B + w_in1 * B + 2 * w * K + w * k +
                                                          (w_in1 + 1) + w * k)
    assert work["csr2"][2] == work["csr2"][0] + 4 * w * k * B
    assert work["forward2"][1] == 132 * w * B
    assert work["forward2"][0] == work["forward2"][2] == 4 * (w * B + w * B + w * K + w * k)
    hw = synth.WORKLOADS["hard_cifar10"]
    N = 1 << 22
    W = N // 32
    hwork = bench.call_work(hw, N)
    assert hwork["hard1"][1] == 63 * 64000 * W
    assert hwork["hard1"][0] == 4 * (21504 * W + 64000 * W + 64000 * 6) + 8 * 64000


def test_byte_wire_layer1_work_and_kernel_names():
    # layer 1 on byte wires: the encoder writes one byte per wire, the
    # lookup forward has no arithmetic (HBM-bound), the one-hot table
    # gradient one add per (node, sample); the call table names the route's
    # kernels
    import types
    import bench
    from paper_2602_07400_gb300 import synth
    wl = synth.WORKLOADS["cifar100"]
    B, d, w_in, w1, K, k = 2048, 3072, 46080, 128000, 64, 6
    f32 = bench.call_work(wl, B, fuse_dy1=True)
    u8 = bench.call_work(wl, B, fuse_dy1=True, bytes1=True)
    assert u8["encode"][0] == B * d + w_in * B < f32["encode"][0]
    assert u8["forward1"][1] == 0 and f32["forward1"][1] == 132 * w1 * B
    assert u8["forward1"][0] == w_in * B + 4 * (w1 * B + w1 * K + w1 * k)
    assert u8["backward1"][1] == w1 * B
    # the fused route moves the per-edge terms in place of dY1
    assert u8["backward1"][2] - u8["backward1"][0] == 4 * w1 * k * B - 4 * w1 * B
    roof = bench.roofline_of("forward1", u8, {"forward1": 0.3}, 152, {}, "none", 6767.1, 2070.0, "measured")
    assert roof["bound"] == "hbm"
    st = types.SimpleNamespace(bytes1=True, through=False, fuse_dy1=True)
    names = bench.kernels_of_step(st)
    assert names["forward1"].startswith("lut_forward_u8_kernel")
    assert names["backward1"].startswith("lut_theta_bytes_kernel")
    st = types.SimpleNamespace(bytes1=True, through=True, fuse_dy1=False)
    assert bench.kernels_of_step(st)["backward1"] == "lut_theta_through_kernel<k, ku, uint8_t>"
    st = types.SimpleNamespace(bytes1=False, through=False, fuse_dy1=False)
    assert bench.kernels_of_step(st)["backward1"] == bench.KERNEL_OF_CALL["backward1"]
    # wire bit rows: one bit per wire and sample (32 words per 1024-sample
    # block), written by the encoder and read by both layer-1 calls
    bw = bench.call_work(wl, B, fuse_dy1=True, bytes1=True, bits1=True)
    xw1 = 4 * w_in * 64            # B = 2048: two blocks of 32 words per row
    assert xw1 * 8 == w_in * B
    assert bw["encode"][0] == B * d + xw1
    assert bw["forward1"][0] == xw1 + 4 * (w1 * B + w1 * K + w1 * k)
    assert bw["backward1"][0] == u8["backward1"][0] - w_in * B + xw1
    assert bw["backward1"][2] - bw["backward1"][0] == u8["backward1"][2] - u8["backward1"][0]
    assert bw["forward2"] == u8["forward2"] and bw["backward1"][1] == w1 * B
    st = types.SimpleNamespace(bytes1=True, bits1=True, through=False, fuse_dy1=True)
    names = bench.kernels_of_step(st)
    assert names["encode"] == "encode_bitrows_kernel" and names["forward1"].startswith("lut_forward_bits_kernel")
    assert "bit rows" in names["backward1"]
    assert bench.route_of_step(st)["layer1_wires"].startswith("bits")


def test_hard_roofline_uses_the_measured_mix_rate():
    # the hard layer's peak is the measured issue rate of its instruction mix
    # (per SM and clock) at the sampled clock; the issue-rate fraction stays
    import bench
    roof = {"achieved": 10.0, "peak": 40.0, "frac": 0.25, "frac_at_sampled_clock": 0.3}
    rates = {"mix": {"lane_ops_per_sm_per_clk": 80.0}}
    got = bench.hard_roofline(roof, rates, 100, {"sm_mhz": 2000.0})
    assert abs(got["peak"] - 80.0 * 100 * 2000e6 / 1e12) < 1e-12
    assert abs(got["frac"] - 10.0 / 16.0) < 1e-12
    assert got["frac_issue_rate"] == 0.25 and got["peak_issue_rate"] == 40.0
    assert abs(got["achieved_per_sm_per_clk"] - 50.0) < 1e-9
    assert "frac_at_sampled_clock" not in got


def test_default_run_is_the_headline_workloads():
    # no --workload: the CIFAR-100-shaped training step and the 2^22-sample
    # hard pass of the CIFAR-10-shaped network, with the extras beside them
    import bench
    from paper_2602_07400_gb300 import synth
    a = bench.parse_args([])
    assert a.workload is None and a.gpus == 1
    assert a.warmup >= 3
    wl = synth.WORKLOADS[bench.HEADLINE_TRAIN]
    assert (wl.batch, wl.widths, wl.k, wl.classes, wl.tau, wl.w_in) == (2048, (128000, 128000), 6, 100, 100.0, 46080)
    wh = synth.WORKLOADS[bench.HEADLINE_HARD]
    assert (wh.batch, wh.widths, wh.k, wh.classes, wh.w_in) == (1 << 22, (64000, 64000), 6, 10, 21504)
    assert set(bench.EXTRAS) == {"mnist", "mnist_k2", "cifar10"}


def test_roofline_object_picks_the_slower_bound():
    import bench
    from paper_2602_07400_gb300 import synth
    wl = synth.WORKLOADS["mnist"]
    work = bench.call_work(wl, 1024)
    per_call = {"backward2": 0.1, "csr2": 0.04}
    roof = bench.roofline_of("backward2", work, per_call, 152, {"sm_mhz": 1035.0}, "no-such-workload",
                             6767.1, 2070.0, "measured")
    assert roof["bound"] == "alu"
    peak = 152 * 128 * 2070e6
    assert abs(roof["achieved"] - 316 * 8000 * 1024 / 1e-4 / 1e12) < 1e-9
    assert abs(roof["frac"] - 316 * 8000 * 1024 / 1e-4 / peak) < 1e-12
    # at half the clock the same time is twice the fraction
    assert abs(roof["frac_at_sampled_clock"] - 2 * roof["frac"]) < 1e-12
    assert roof["traffic"] is None and roof["traffic_over_algorithmic"] is None
    hroof = bench.roofline_of("csr2", work, per_call, 152, {}, "x", 6767.1, 2070.0, "measured")
    assert hroof["bound"] == "hbm"
    assert abs(hroof["achieved"] - work["csr2"][0] / 4e-5 / 1e9) < 1e-6
    names = ["encode", "forward1", "forward2", "head", "backward2", "csr2", "backward1"]
    frac = bench.step_hbm_fraction(wl, 1024, work, names, 0.2, 6767.1)
    assert frac["moved_over_algorithmic"] > 1.0
    assert frac["frac_hbm_survey"] > frac["frac_hbm"]


def test_step_bytes_follow_the_survey_formula():
    # C3 (CIFAR-10-shaped, B = 1024): ~2.64 GB per step for the two layers
    # and the head with one gradient row per node, plus the encoder (3.1 MB
    # of pixels in, 88.1 MB of bits out); the per-class rows save the head's
    # dY write and the layer-2 backward's dY read (2 x 262 MB) less the
    # C x B rows
    import bench
    from paper_2602_07400_gb300 import synth
    wl = synth.WORKLOADS["cifar10"]
    sb = bench.step_bytes(wl, 1024)
    enc = 1024 * 3072 + 4 * 21504 * 1024
    assert abs((sb["survey"] - enc) / 1e9 - 2.64) < 0.005, sb
    wB = 4 * 64000 * 1024
    assert abs((sb["survey"] - sb["design"]) - (2 * wB - 4 * (3 * 1024 * 10 + 1024))) < 1
    # the per-call algorithmic bytes of the unfused step add up to the
    # design total
    work = bench.call_work(wl, 1024)
    names = ["encode", "forward1", "forward2", "head", "backward2", "csr2", "backward1"]
    assert abs(sum(work[n][0] for n in names) / sb["design"] - 1) < 1e-3
