#!/usr/bin/env python3
"""Throughput of the LUT-network hot path on GB300 (one JSON line on rank 0).

A step is one pass of the whole hot path over one batch of synthetic input:
the soft training step (thermometer encode, two LUT forwards, group-sum head
with cross-entropy, two LUT backwards with the CSR input-gradient
reduction) followed by the hard evaluation of the same batch (table
binarization, encode + pack, hard layer 1, hard layer 2 with the fused
popcount head and argmax).  ``value`` is the training throughput (samples
per second through the fwd+bwd part); the hard part is reported in the
``hard`` object.  L2 is flushed between steps (a 512 MB write outside the
timed events), so every step starts cold.  The timed loop replays the step as
CUDA graphs captured once (no host work between launches); the per-call
split comes from eager steps with an event after every call.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--workload mnist]
  python bench.py --impl reference ...   # the CPU oracle on the same workload

Multi-GPU (torchrun, one process per GPU): every rank trains its own batch
(weak scaling, no data-path collective); the job's time is the max over
ranks and ``value`` sums the samples of all ranks.
"""
from __future__ import annotations

import argparse
import hashlib
import json
import os
import re
import statistics
import subprocess
import sys
import tempfile
import time

import numpy as np
import torch

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

from paper_2602_07400_gb300 import synth  # noqa: E402

METRIC = "LUT train samples/s (fwd+bwd) and hard bit-packed MSamples/s; % of roofline"
FP32_LANES_PER_SM = 128
# the paper's own figures for a workload of the same shape, on its hardware
# (context only, not a target: another machine and its own timing protocol)
PAPER_CONTEXT = {
    "hard_mnist_w4000": "paper, hardware evaluation table: RTX 3090 bit-packed forward of the w=4000 MNIST "
                        "network, batch 1024: 8.66 MSamples/s (RTX 2080 Ti 6.98)",
    "hard_mnist_w4000_4m": "paper, hardware evaluation table: RTX 3090 bit-packed forward of the w=4000 MNIST "
                           "network, batch 1024: 8.66 MSamples/s; FPGA max-throughput mode ~126 MSamples/s",
}
SMI_FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")


def parse_args():
    p = argparse.ArgumentParser()
    p.add_argument("--gpus", type=int, default=1)
    p.add_argument("--steps", type=int, default=400)
    p.add_argument("--warmup", type=int, default=20)
    p.add_argument("--impl", choices=["ours", "reference"], default="ours")
    p.add_argument("--workload", default="mnist", choices=sorted(synth.WORKLOADS))
    p.add_argument("--node", default="soft", choices=["soft", "st"],
                   help="LightLUT node form of the training step: soft, or straight-through hard")
    p.add_argument("--no-cpu-baseline", action="store_true")
    p.add_argument("--no-e2e", action="store_true")
    p.add_argument("--no-graph", action="store_true",
                   help="time eager launches instead of CUDA-graph replays of the step")
    p.add_argument("--profile", action="store_true",
                   help="plain timed loop only (for ncu launch lists)")
    p.add_argument("--batch", type=int, default=0,
                   help="override the workload's batch (smaller cases for ncu captures)")
    return p.parse_args()


def peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(path):
        with open(path) as f:
            m = json.load(f)
        return float(m["hbm_gbs"]), float(m.get("sm_max_mhz", 2070.0)), "measured"
    return 6800.0, 2070.0, "fallback"


# ------------------------------------------------------------- clocks --

class ClockSampler:
    def __init__(self, index: int, period_ms: int = 100):
        self.index, self.period = index, period_ms
        self.proc = None
        self.path = None

    def start(self):
        try:
            fd, self.path = tempfile.mkstemp(suffix=".csv")
            os.close(fd)
            self.out = open(self.path, "w")
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--id={self.index}", f"--query-gpu={SMI_FIELDS}",
                 "--format=csv,noheader,nounits", f"-lms", str(self.period)],
                stdout=self.out, stderr=subprocess.DEVNULL)
        except (OSError, FileNotFoundError):
            self.proc = None
        self.t0 = time.time()

    def stop(self):
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": [], "samples": 0,
                    "note": "nvidia-smi unavailable"}
        time.sleep(0.25)
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        self.out.close()
        sm, mx, pw, reasons = [], [], [], set()
        names = ["active", "hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        with open(self.path) as f:
            for line in f:
                parts = [p.strip() for p in line.split(",")]
                if len(parts) < 9:
                    continue
                try:
                    sm.append(float(parts[1]))
                    mx.append(float(parts[2]))
                    pw.append(float(parts[3]))
                except ValueError:
                    continue
                for name, val in zip(names[1:], parts[5:9]):
                    if val.lower().startswith("active"):
                        reasons.add(name)
        os.unlink(self.path)
        return {"sm_mhz": statistics.median(sm) if sm else None,
                "sm_max_mhz": max(mx) if mx else None,
                "power_w_max": max(pw) if pw else None,
                "reasons": sorted(reasons), "samples": len(sm)}


# ------------------------------------------------- cross-rank helpers --

def max_over_ranks(values, device):
    """Element-wise max of per-rank timings (the job is as slow as its
    slowest rank)."""
    import torch.distributed as dist
    t = torch.tensor([float(v) for v in values], dtype=torch.float64, device=device)
    if dist.is_available() and dist.is_initialized() and dist.get_world_size() > 1:
        dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return [float(v) for v in t.tolist()]


def job_rate(world: int, samples_per_rank_step: int, steps: int, max_ms: float) -> float:
    """Whole-job samples/s: every rank's samples over the slowest rank's time."""
    return world * samples_per_rank_step * steps / (max_ms * 1e-3)


# ------------------------------------------------------ work per call --

def call_work_routed(wl, B):
    """Work of the calls of a routed training step: the routing calls count
    their HBM bytes (each slot's Kc candidate rows are gathered from the
    layer input, which stays in L2, so the gathered bytes are not HBM
    traffic) and one FMA per (candidate, sample); the LUT calls read the
    slot rows through the identity connectivity."""
    K, k, Kc = wl.K, wl.k, wl.Kc
    w1, w2 = wl.widths
    win, d, C = wl.w_in, wl.d, wl.classes
    s1, s2 = w1 * k, w2 * k
    f = 4
    return {
        # the encoder's wires are bytes in the routed step (layer 1 gathers them)
        "encode": (B * d + win * B, 0),
        "route1": (win * B + f * (s1 * B + 2 * s1 * Kc), Kc * s1 * B),
        "forward1": (f * (s1 * B + w1 * B + w1 * K + w1 * k), (2 * (K - 1) + k) * w1 * B),
        "route2": (f * (w1 * B + s2 * B + 2 * s2 * Kc), Kc * s2 * B),
        "forward2": (f * (s2 * B + w2 * B + w2 * K + w2 * k), (2 * (K - 1) + k) * w2 * B),
        "head": (f * (w2 * B + 4 * B * C), 0),
        "backward2": (f * (s2 * B + C * B + s2 * B + 2 * w2 * K + w2 * k), (4 * (K - 1) + K) * w2 * B),
        "route_bwd2": (f * (w1 * B + 2 * s2 * B + w1 * B + 3 * s2 * Kc), 2 * Kc * s2 * B),
        "backward1": (f * (s1 * B + w1 * B + s1 * B + 2 * w1 * K + w1 * k), (4 * (K - 1) + K) * w1 * B),
        "route_bwd1": (win * B + f * (s1 * B + 2 * s1 * Kc), Kc * s1 * B),
        "binarize": (f * (w1 * K + w2 * K) + 8 * (w1 + w2), 0),
        "pack": (B * d + f * win * ((B + 31) // 32), 0),
        "hard1": (f * (win * ((B + 31) // 32) + w1 * ((B + 31) // 32) + w1 * k) + 8 * w1,
                  (K - 1) * w1 * ((B + 31) // 32)),
        "hard2": (f * (w1 * ((B + 31) // 32) + w2 * k + B * C * 2 + B) + 8 * w2, (K - 1) * w2 * ((B + 31) // 32)),
    }


def call_work(wl, B, fuse_dy1=False):
    """Algorithmic work of each library call of one step on a batch of B:
    (bytes, fp32 or logic ops).  Ops follow the lerp-tree counts: forward
    2(2^k-1)+k per (node, sample); backward with input gradient
    4(2^k-1)+2^k; backward without it 2(2^k-1)+2^k; hard layer 2^k-1 LOP3
    per (node, 32-sample word)."""
    K, k = wl.K, wl.k
    w1, w2 = wl.widths
    win, d, b, C = wl.w_in, wl.d, wl.b, wl.classes
    W = (B + 31) // 32
    f = 4
    return {
        "encode": (B * d + f * win * B, 0),
        "forward1": (f * (win * B + w1 * B + w1 * K + w1 * k), (2 * (K - 1) + k) * w1 * B),
        "forward2": (f * (w1 * B + w2 * B + w2 * K + w2 * k), (2 * (K - 1) + k) * w2 * B),
        "head": (f * (w2 * B + 4 * B * C), 0),
        # layer 2: reads Y1 and the per-class gradient rows, writes dtheta and
        # the per-edge input-gradient terms
        "backward2": (f * (w1 * B + C * B + w2 * k * B + 2 * w2 * K + w2 * k), (4 * (K - 1) + K) * w2 * B),
        # layer 1 (fused form): reads the encoder bits and layer 2's per-edge
        # terms (its output gradient, reduced through the CSR map in the
        # kernel); unfused form: the CSR reduction of those terms into dY1
        # ("csr2"), then the dtheta-only backward reading dY1
        "backward1": (f * (win * B + w2 * k * B + 2 * w1 * K + w1 * k + w1 + w2 * k), (2 * (K - 1) + K) * w1 * B)
        if fuse_dy1 else (f * (win * B + w1 * B + 2 * w1 * K + w1 * k), (2 * (K - 1) + K) * w1 * B),
        "csr2": (f * (w2 * k * B + w1 * B + w1 + 1 + w2 * k), 0),
        "binarize": (f * (w1 * K + w2 * K) + 8 * (w1 + w2), 0),
        "pack": (B * d + f * win * W, 0),
        "hard1": (f * (win * W + w1 * W + w1 * k) + 8 * w1, (K - 1) * w1 * W),
        "hard2": (f * (w1 * W + w2 * k + B * C * 2 + B) + 8 * w2, (K - 1) * w2 * W),
    }


# DRAM traffic per launch of the roofline kernel, dram__bytes_read.sum +
# dram__bytes_write.sum from one ncu capture, keyed by workload
# and call.  Valid only for the kernel source it was taken on: the SHA-256 of
# the source file's code (comments and blank space removed) is recorded, and
# any later change of the code reports null.
TRAFFIC = {
    ("mnist", "backward2"): {
        "bytes": 59.670016e6 + 147.641856e6, "source": "lut_soft.cu",
        "sha256": "180fc79502da4e837de466268e4dd9af96f7da65e286f6b8dce737f118e99f43",
        "note": "ncu capture of this workload"},
    ("hard_cifar10", "hard1"): {
        "bytes": 16 * (1.209681e9 + 2.054784e9), "source": "hard.cu",
        "sha256": "f9bed6fc20215df71b5e12eebae1c94762286b3c7b941dea9a2ff948bfb9ed3c",
        "note": "ncu capture at 2^18 samples, scaled x16 to 2^22 by the words processed"},
}


def code_digest(path: str) -> str:
    """SHA-256 of a C++/CUDA source with its comments and blank space
    removed, so that edits of the comments keep a capture valid."""
    with open(path, encoding="utf-8") as f:
        src = f.read()
    src = re.sub(r"/\*.*?\*/", " ", src, flags=re.S)
    src = re.sub(r"//[^\n]*", " ", src)
    src = " ".join(src.split())
    return hashlib.sha256(src.encode()).hexdigest()


def kernel_traffic(workload: str, call: str):
    """(bytes per launch, note) when the capture matches the current source, else (None, why)."""
    t = TRAFFIC.get((workload, call))
    if t is None:
        return None, "no capture for this workload"
    path = os.path.join(ROOT, "paper_2602_07400_gb300", "csrc", t["source"])
    try:
        digest = code_digest(path)
    except OSError:
        return None, "kernel source not found"
    if digest != t["sha256"]:
        return None, f"{t['source']} changed since the capture"
    return t["bytes"], t["note"]


KERNEL_OF_CALL = {
    "encode": "encode_soft_kernel", "forward1": "lut_forward_staged_kernel<k>",
    "forward2": "lut_forward_staged_kernel<k>", "head": "head_* (3 kernels)",
    "backward2": "lut_backward_node_kernel<k, dx, dY rows>",
    "backward1": "lut_backward_theta_kernel<k>", "csr2": "csr_reduce_kernel",
    "binarize": "binarize_kernel (x2)", "pack": "pack_bits_kernel", "hard1": "hard_layer_staged_kernel<k>",
    "hard2": "hard_head_staged_kernel<k> + argmax_kernel",
    "route1": "route_forward_vec_kernel<KC>", "route2": "route_forward_vec_kernel<KC>",
    "route_bwd2": "route_dr_kernel + route_dx_kernel", "route_bwd1": "route_dr_kernel<KC> (byte rows)",
}


# --------------------------------------------------------------- ours --

def dist_env():
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return world, rank, local


def run_ours(args):
    import paper_2602_07400_gb300 as bl
    from paper_2602_07400_gb300.pipeline import HardInfer, Network, RoutedNetwork, RoutedTrainStep, TrainStep

    world, rank, local = dist_env()
    torch.cuda.set_device(local)
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
    bl.load()
    wl = synth.WORKLOADS[args.workload]
    if args.batch:
        wl = synth.Workload(wl.name, args.batch, wl.d, wl.classes, wl.sigma, wl.thresholds,
                            wl.widths, wl.k, wl.tau)
    hard_only = wl.name.startswith("hard_")
    B = wl.batch
    if wl.Kc:
        rnet = RoutedNetwork(*synth.routed_network(wl, seed=0), wl.w_in)
        net = rnet.snap()                # the hard pass evaluates the discretized network
    else:
        conn1, th1, conn2, th2 = synth.network(wl, seed=0)
        net = Network(conn1, th1, conn2, th2, wl.w_in)
    x_gen, lab_gen = synth.blob_batch(B, wl.d, wl.classes, wl.sigma, seed=1000 + rank,
                                      device="cuda" if hard_only else "cpu")
    st = None
    if not hard_only:
        if wl.Kc:
            st = RoutedTrainStep(rnet, B, wl.d, wl.thresholds, wl.classes, wl.tau, node=args.node)
        else:
            st = TrainStep(net, B, wl.d, wl.thresholds, wl.classes, wl.tau, node=args.node)
        st.load(x_gen.cuda(), lab_gen.cuda())
    hi = HardInfer(net, B, wl.d, wl.thresholds, wl.classes)
    if st is not None:
        hi.x = st.x                      # the hard pass evaluates the same batch
    else:
        hi.x.copy_(x_gen)
    del x_gen
    flush = torch.empty(512 << 20, dtype=torch.uint8, device="cuda")
    stream = torch.cuda.current_stream()

    def step(mark):
        if st is not None:
            st.run(mark=mark)
            mark("train_end")
        hi.binarize(mark=mark)
        hi.run(mark=mark)

    for _ in range(args.warmup):
        flush.fill_(1)
        step(lambda n: None)
    torch.cuda.synchronize()

    K = args.steps
    use_graph = not (args.no_graph or args.profile)

    def eager_steps(n):
        """n eager steps with a CUDA event after every library call:
        per-call durations and per-step (train, hard) sums."""
        marks = []
        for _ in range(n):
            flush.fill_(1)
            lst = []
            marks.append(lst)

            def mark(name, lst=lst):
                ev = torch.cuda.Event(enable_timing=True)
                ev.record(stream)
                lst.append((name, ev))
            mark("start")
            step(mark)
        torch.cuda.synchronize()
        calls, train_ms, hard_ms = {}, [], []
        for lst in marks:
            prev = lst[0][1]
            t_train = 0.0
            t_total = 0.0
            for name, ev in lst[1:]:
                dt = prev.elapsed_time(ev)
                prev = ev
                if name == "train_end":
                    t_train = t_total
                    continue
                calls.setdefault(name, []).append(dt)
                t_total += dt
            train_ms.append(t_train)
            hard_ms.append(t_total - t_train)
        return calls, train_ms, hard_ms

    if use_graph:
        # the step as two CUDA graphs (training fwd+bwd; hard pass with its
        # binarization), replayed in the timed loop
        g_train = st.capture() if st is not None else None
        g_hard = hi.capture(binarize=True)
        for _ in range(3):
            flush.fill_(1)
            if g_train is not None:
                g_train.replay()
            g_hard.replay()
        torch.cuda.synchronize()

    clock = ClockSampler(local)
    if world > 1:
        torch.distributed.barrier()
    torch.cuda.synchronize()
    clock.start()
    wall0 = time.perf_counter()
    if use_graph:
        evs = []
        for _ in range(K):
            flush.fill_(1)
            e = [torch.cuda.Event(enable_timing=True) for _ in range(3)]
            e[0].record(stream)
            if g_train is not None:
                g_train.replay()
            e[1].record(stream)
            g_hard.replay()
            e[2].record(stream)
            evs.append(e)
        torch.cuda.synchronize()
        train_ms = [e[0].elapsed_time(e[1]) for e in evs]
        hard_ms = [e[1].elapsed_time(e[2]) for e in evs]
    else:
        calls, train_ms, hard_ms = eager_steps(K)
    wall = time.perf_counter() - wall0
    if world > 1:
        torch.distributed.barrier()
    clocks = clock.stop()
    assert bl.bitlogic_device_error() == 0
    train_sum, hard_sum = max_over_ranks([sum(train_ms), sum(hard_ms)], "cuda")
    eager_ms = None
    if use_graph:
        # per-call split (and the roofline kernel's duration) from eager steps
        # with an event after every call, outside the timed loop
        calls, tr_e, hd_e = eager_steps(max(3, min(K, 100)))
        eager_ms = {"train": float(np.mean(tr_e)), "hard": float(np.mean(hd_e))}

    launches = K * (hi.kernels_per_binarize + hi.kernels_per_run)
    if st is not None:
        launches += K * st.kernels_per_run

    result = None
    if rank == 0:
        hbm, sm_max, peak_kind = peaks()
        work = call_work_routed(wl, B) if wl.Kc else call_work(wl, B, fuse_dy1=st.fuse_dy1 if st is not None else False)
        per_call_ms = {n: float(np.mean(v)) for n, v in calls.items()}
        ms_step_train = train_sum / K
        ms_step_hard = hard_sum / K
        # roofline of the dominant single-kernel call
        single = {n: t for n, t in per_call_ms.items() if n not in ("head", "binarize", "hard2", "route_bwd2")}
        dom = max(single, key=single.get)
        byts, ops = work[dom]
        t_s = per_call_ms[dom] * 1e-3
        fp32_peak = 152 * FP32_LANES_PER_SM * sm_max * 1e6
        t_hbm, t_alu = byts / (hbm * 1e9), ops / fp32_peak
        if t_alu >= t_hbm:
            unit = ("Tops/s (integer mux lane-ops against the issue rate)" if dom.startswith("hard")
                    else "Tops/s (fp32 pipe lane-ops)")
            roof = {"bound": "alu", "achieved": ops / t_s / 1e12, "peak": fp32_peak / 1e12, "unit": unit}
        else:
            roof = {"bound": "hbm", "achieved": byts / t_s / 1e9, "peak": hbm, "unit": "GB/s"}
        roof["frac"] = roof["achieved"] / roof["peak"]
        traffic, traffic_note = kernel_traffic(wl.name, dom)
        roof.update({"traffic": traffic, "traffic_source": traffic_note, "kernel": KERNEL_OF_CALL[dom], "call": dom,
                     "ms_per_launch": per_call_ms[dom], "algorithmic_bytes": byts,
                     "algorithmic_ops": ops, "peak_source": f"{peak_kind} (HBM), "
                     f"152 SMs x {FP32_LANES_PER_SM} lanes x {sm_max:.0f} MHz (alu: one issue per lane "
                     f"and clock)"})
        calls_out = {}
        for n, t in per_call_ms.items():
            b_, o_ = work[n]
            calls_out[n] = {"ms": round(t, 5), "GB/s": round(b_ / (t * 1e-3) / 1e9, 1),
                            "Tops/s": round(o_ / (t * 1e-3) / 1e12, 2) if o_ else None}
        value = job_rate(world, B, K, train_sum if st is not None else hard_sum)
        result = {
            "metric": METRIC,
            "value": value,
            "unit": "samples/s",
            "n_gpus": world,
            "steps": K,
            "warmup": args.warmup,
            "ms_per_step": ms_step_train if st is not None else ms_step_hard,
            "higher_is_better": True,
            "scaling": "weak",
            "vs_baseline": None,
            "dtype": "f32",
            "data": "synthetic (seeded class-conditional Gaussian blobs, MNIST/CIFAR shapes; random-init tables)",
            "config": {"workload": wl.name, "batch_per_gpu": B, "d": wl.d, "thresholds": list(wl.thresholds),
                       "widths": list(wl.widths), "k": wl.k, "classes": wl.classes, "tau": wl.tau,
                       "routing": f"learnable, {wl.Kc} candidates per slot" if wl.Kc else "fixed (random-unique)",
                       "node": "LightLUT " + ("soft" if args.node == "soft" else "straight-through hard"),
                       "l2": "flushed between steps (512 MB write outside the timed events)",
                       "parallelism": f"dp{world} (independent batches, no collective)"},
            "hard": {"value": job_rate(world, B, K, hard_sum) / 1e6, "unit": "MSamples/s",
                     "ms_per_batch": ms_step_hard, "batch": B,
                     "includes": "binarize + encode/pack + 2 hard layers + popcount head + argmax"},
            "ms_per_step_total": ms_step_train + ms_step_hard,
            "timing": ("CUDA-graph replays of the step (training fwd+bwd graph, hard-pass graph), CUDA events "
                       "around each replay; per-call split from eager steps with an event after every call"
                       if use_graph else "eager launches, CUDA events after every library call"),
            **({"eager_ms_per_step": eager_ms} if eager_ms else {}),
            **({"context": PAPER_CONTEXT[wl.name]} if wl.name in PAPER_CONTEXT else {}),
            "calls": calls_out,
            "roofline": roof,
            "gpu_launches": launches,
            "clocks": clocks,
            "wall_s_timed_loop": wall,
        }
    if st is not None and not args.profile:
        # the AdamW update of both layers' logits (not part of `value`, which
        # is the fwd+bwd step): timed on its own from the last gradients
        upd = time_update(st, max(3, min(args.steps, 50)))
        if result is not None:
            n_par = int(st.net.theta1.numel() + st.net.theta2.numel())
            if wl.Kc:
                n_par += int(st.net.r1.numel() + st.net.r2.numel())
            result["optimizer"] = {"ms_per_update": upd,
                                   "kernel": f"adamw_vec_kernel (x{4 if wl.Kc else 2})",
                                   "algorithmic_bytes": 28 * n_par,
                                   "GB/s": 28 * n_par / (upd * 1e-3) / 1e9,
                                   "settings": "AdamW beta (0.9, 0.999), eps 1e-8, lr 0.01, wd 0"}
    if st is not None and world > 1 and not args.profile:
        # the data-parallel exchange of a training step (all-reduce of the
        # gradients before the update), timed on its own: the fwd+bwd step
        # above has no collective
        from paper_2602_07400_gb300.pipeline import allreduce_gradients
        grads = st.gradients()
        for _ in range(3):
            allreduce_gradients(grads)
        torch.cuda.synchronize()
        torch.distributed.barrier()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record()
        for _ in range(20):
            allreduce_gradients(grads)
        e1.record()
        torch.cuda.synchronize()
        ms_x = max_over_ranks([e0.elapsed_time(e1) / 20], "cuda")[0]
        if result is not None:
            result["dp_exchange"] = {"ms": ms_x, "collective": "NCCL all-reduce (sum) of the gradients, then / N",
                                     "bytes_per_rank": int(sum(g.numel() * 4 for g in grads))}
    if not args.profile and rank == 0:
        result["fit"] = time_quantile_fit(wl, flush)
        result["pipe_rates"] = measure_pipe_rates()
        if result["roofline"]["call"] in ("hard1", "hard2"):
            result["roofline"]["integer_pipes"] = integer_pipe_fraction(result["roofline"], result["pipe_rates"])
    if not args.profile and not args.no_e2e:
        e2e = run_e2e(args, st, hi, wl, B, use_graph)
        if result is not None:
            result["e2e"] = e2e["train"] if st is not None else e2e["hard"]
            result["hard"]["e2e"] = e2e["hard"]
    if world > 1:
        torch.distributed.barrier()
        torch.distributed.destroy_process_group()
    return result


# training split sizes of the datasets the workloads stand in for
SPLIT_SAMPLES = {784: 60000, 3072: 50000}


def time_quantile_fit(wl, flush, iters: int = 20):
    """The quantile thermometer fit's device pass (the pixel histogram) over a
    training split of the workload's shape, L2 flushed before every call."""
    import paper_2602_07400_gb300 as bl
    n_samples = SPLIT_SAMPLES.get(wl.d, 50000)
    x, _ = synth.blob_batch(n_samples, wl.d, wl.classes, wl.sigma, seed=5000, device="cuda")
    hist = torch.zeros(256, dtype=torch.int64, device="cuda")
    for _ in range(3):
        bl.bitlogic_pixel_histogram(x, hist)
    ms = []
    for _ in range(iters):
        flush.fill_(2)
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record()
        bl.bitlogic_pixel_histogram(x, hist)
        e1.record()
        ms.append((e0, e1))
    torch.cuda.synchronize()
    t = float(np.mean([a.elapsed_time(b) for a, b in ms]))
    hbm, _, _ = peaks()
    gbs = x.numel() / (t * 1e-3) / 1e9
    thr = bl.bitlogic_quantile_thresholds(hist, wl.b)
    return {"kernel": "pixel_histogram_kernel", "split": f"{n_samples} x {wl.d} uint8 (a training split of the "
            f"workload's shape)", "ms": t, "GB/s": gbs, "frac_hbm": gbs / hbm,
            "thresholds_b": [int(v) for v in thr]}


def measure_pipe_rates(iters: int = 2048, reps: int = 5) -> dict:
    """Sustained issue rates of the pipes the kernels run on, from the
    library's throughput probe (independent chains of one instruction kind
    over 4 blocks of 256 threads per SM): LOP3 (logic pipe, the hard mux
    tree's upper levels), IMAD (FMA pipe, its level 0) and FFMA (FMA pipe,
    the soft kernels).  Median of `reps` launches, CUDA events."""
    import paper_2602_07400_gb300 as bl
    n = bl.bitlogic_issue_probe_threads()
    sms = n // (4 * 256)
    sink = torch.empty(n, dtype=torch.int32, device="cuda")
    ops = n * iters * bl.bitlogic_issue_probe_ops_per_iter()
    _, sm_max, _ = peaks()
    out = {"sms": sms, "clock_mhz_assumed": sm_max,
           "probe": "independent dependency chains, 4 x 256 threads per SM, median of 5 launches"}
    for kind in ("lop3", "imad", "ffma"):
        bl.bitlogic_issue_probe(kind, iters, sink)
        evs = []
        for _ in range(reps):
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record()
            bl.bitlogic_issue_probe(kind, iters, sink)
            e1.record()
            evs.append((e0, e1))
        torch.cuda.synchronize()
        t = float(np.median([a.elapsed_time(b) for a, b in evs]))
        rate = ops / (t * 1e-3)
        out[kind] = {"T_lane_ops_s": round(rate / 1e12, 3),
                     "lane_ops_per_sm_per_clk": round(rate / (sms * sm_max * 1e6), 1)}
    return out


def integer_pipe_fraction(roof: dict, rates: dict) -> dict:
    """The hard layer's mux operations against the measured integer ceiling:
    a mix of IMAD (FMA pipe) and LOP3 (logic pipe) can at best keep both
    pipes busy, so the ceiling is the sum of their measured rates (below the
    issue rate the main roofline uses)."""
    peak = rates["imad"]["T_lane_ops_s"] + rates["lop3"]["T_lane_ops_s"]
    return {"peak": round(peak, 3), "unit": "T lane-ops/s", "frac": roof["achieved"] / peak,
            "source": "issue probe: IMAD + LOP3 (mux) rates measured in this run"}


def time_update(st, iters: int) -> float:
    """Mean ms of one AdamW update of both layers (CUDA events on the launching stream)."""
    for _ in range(3):
        st.update()
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record()
    for _ in range(iters):
        st.update()
    e1.record()
    torch.cuda.synchronize()
    return e0.elapsed_time(e1) / iters


def run_e2e(args, st, hi, wl, B, use_graph=True):
    """The same metric end to end through the public API: every step copies
    its batch from pinned host memory and its result (loss, or predictions)
    back.  With graphs, ``pipeline.Prefetcher`` overlaps the copy of the
    next batch with the current step (two input buffers, a copy stream);
    without, the copy, the step and the read-back run in sequence."""
    from paper_2602_07400_gb300.pipeline import Prefetcher
    world, rank, _ = dist_env()
    x_host, lab_host = synth.blob_batch(B, wl.d, wl.classes, wl.sigma, seed=2000 + rank)
    x_host = x_host.pin_memory()
    lab_host = lab_host.pin_memory()
    loss_host = torch.empty(1, dtype=torch.float32).pin_memory()
    pred_host = torch.empty(B, dtype=torch.int32).pin_memory()
    K = max(1, args.steps)
    out = {}

    def timed(pf, host, res, eager):
        if pf is None:
            for _ in range(3):
                eager()
            torch.cuda.synchronize()
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record()
            for _ in range(K):
                eager()
            e1.record()
            torch.cuda.synchronize()
            return max_over_ranks([e0.elapsed_time(e1)], "cuda")[0]
        for _ in range(3):
            pf.prefetch(host)
            pf.run(res)
        torch.cuda.synchronize()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record()
        pf.start()
        pf.prefetch(host)
        for i in range(K):
            if i + 1 < K:
                pf.prefetch(host)   # batch i + 1 streams in while step i runs
            pf.run(res)
        e1.record()
        torch.cuda.synchronize()
        return max_over_ranks([e0.elapsed_time(e1)], "cuda")[0]

    if st is not None:
        def eager_train():
            st.load(x_host, lab_host, non_blocking=True)
            st.run()
            loss_host.copy_(st.loss, non_blocking=True)
        pf = Prefetcher(st, ("x", "labels"), "loss") if use_graph else None
        ms = timed(pf, {"x": x_host, "labels": lab_host}, loss_host, eager_train)
        out["train"] = {"value": job_rate(world, B, K, ms), "unit": "samples/s",
                        "h2d_bytes_per_step": x_host.numel() + 4 * lab_host.numel(),
                        "d2h_bytes_per_step": 4, "overlap": bool(use_graph)}

    def eager_hard():
        hi.x.copy_(x_host, non_blocking=True)
        hi.binarize()
        hi.run()
        pred_host.copy_(hi.pred, non_blocking=True)
    pf = Prefetcher(hi, ("x",), "pred", capture=lambda: hi.capture(binarize=True)) if use_graph else None
    ms = timed(pf, {"x": x_host}, pred_host, eager_hard)
    out["hard"] = {"value": job_rate(world, B, K, ms) / 1e6, "unit": "MSamples/s",
                   "h2d_bytes_per_step": x_host.numel(), "d2h_bytes_per_step": 4 * B, "overlap": bool(use_graph)}
    return out


# -------------------------------------------------- oracle (CPU) legs --

_NETWORKS = {}


def _network(wl):
    """The workload's network (drawn once per process)."""
    if wl.name not in _NETWORKS:
        _NETWORKS[wl.name] = synth.routed_network(wl, seed=0) if wl.Kc else synth.network(wl, seed=0)
    return _NETWORKS[wl.name]


def oracle_train_rate(wl, samples: int, seed: int = 0, node: str = "soft"):
    import oracle
    x, lab = synth.blob_batch(samples, wl.d, wl.classes, wl.sigma, seed=3000 + seed)
    if wl.Kc:
        params = _network(wl)
        t0 = time.perf_counter()
        oracle.routed_train_step(x.numpy(), lab.numpy(), wl.thresholds, *params, wl.classes, wl.tau, node=node)
        return samples / (time.perf_counter() - t0)
    conn1, th1, conn2, th2 = _network(wl)
    t0 = time.perf_counter()
    oracle.train_step(x.numpy(), lab.numpy(), wl.thresholds, conn1, th1, conn2, th2,
                      wl.classes, wl.tau, node=node)
    return samples / (time.perf_counter() - t0)


def oracle_hard_rate(wl, samples: int, seed: int = 0):
    import oracle
    conn1, th1, conn2, th2 = synth.network(wl, seed=0) if wl.Kc else _network(wl)
    t1, t2 = oracle.binarize_tables(th1), oracle.binarize_tables(th2)
    x, _ = synth.blob_batch(samples, wl.d, wl.classes, wl.sigma, seed=4000 + seed)
    t0 = time.perf_counter()
    oracle.hard_infer(x.numpy(), wl.thresholds, conn1, t1, conn2, t2, wl.classes)
    return samples / (time.perf_counter() - t0)


def calibrated(rate_fn, wl, budget_s: float, lo: int, hi: int):
    r0 = rate_fn(wl, lo)
    n = int(min(hi, max(lo, r0 * budget_s)))
    n = max(lo, (n // lo) * lo)
    return rate_fn(wl, n, seed=1), n


def cpu_baseline(wl, budget_s=12.0, node="soft"):
    import oracle
    hard_only = wl.name.startswith("hard_")
    cores = oracle.max_threads()
    out = {}
    if not hard_only:
        r, n = calibrated(lambda w_, n_, seed=0: oracle_train_rate(w_, n_, seed, node), wl, budget_s, 4, wl.batch)
        out = {"value": r, "unit": "samples/s", "cores": cores, "kind": "oracle",
               "sample": f"train step (fwd+bwd) on {n} of the {wl.batch} samples of a batch, "
                         f"full network, fp64, OpenMP over independent outputs"}
    rh, nh = calibrated(oracle_hard_rate, wl, budget_s / 2, 32, 1 << 16)
    hard = {"value": rh / 1e6, "unit": "MSamples/s", "cores": cores, "kind": "oracle",
            "sample": f"hard pass (encode+pack, 2 layers, popcount head) on {nh} samples"}
    return out, hard


def run_reference(args):
    world, rank, _ = dist_env()
    if rank != 0:
        return None
    import oracle
    wl = synth.WORKLOADS[args.workload]
    hard_only = wl.name.startswith("hard_")
    fn = oracle_hard_rate if hard_only else (lambda w_, n_, seed=0: oracle_train_rate(w_, n_, seed, args.node))
    lo = 32 if hard_only else 2
    # size one step so that the whole run (warm-up and timed steps) takes
    # about two minutes of oracle work, at most 1.5 s per step; the rate is
    # calibrated on a sample large enough to amortise the per-call set-up
    per_step_s = min(1.5, 120.0 / max(1, args.steps + args.warmup))
    r0 = fn(wl, min(wl.batch, 4096 if hard_only else 64))
    n = max(lo, int(r0 * per_step_s) // lo * lo)
    n = min(n, wl.batch)
    for i in range(args.warmup):
        fn(wl, lo, seed=100 + i)
    tot_s, tot_n = 0.0, 0
    for i in range(args.steps):
        r = fn(wl, n, seed=i)
        tot_s += n / r
        tot_n += n
    value = tot_n / tot_s
    unit = "samples/s"
    if hard_only:
        value /= 1e6
        unit = "MSamples/s"
    cores = oracle.max_threads()
    return {
        "impl": "reference", "metric": METRIC, "value": value, "unit": unit, "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1e3 * tot_s / max(1, args.steps),
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
        "data": "synthetic", "config": {"workload": wl.name, "batch_per_gpu": wl.batch},
        "cpu_baseline": {"value": value, "unit": unit, "cores": cores, "kind": "oracle",
                         "sample": f"{n} samples of the workload per step (the plain C oracle, "
                                   f"{'hard pass' if hard_only else 'train fwd+bwd'})"},
        "e2e": {"value": value, "unit": unit, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }


def main():
    args = parse_args()
    if args.impl == "reference":
        res = run_reference(args)
        if res is not None:
            print(json.dumps(res), flush=True)
        return
    res = run_ours(args)
    if res is None:
        return
    if not args.profile and not args.no_cpu_baseline:
        wl = synth.WORKLOADS[args.workload]
        cb, cb_hard = cpu_baseline(wl, node=args.node)
        if cb:
            res["cpu_baseline"] = cb
        res["hard"]["cpu_baseline"] = cb_hard
    print(json.dumps(res), flush=True)


if __name__ == "__main__":
    main()
