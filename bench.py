#!/usr/bin/env python3
"""Throughput of the LUT-network hot path on GB300 (one JSON line on rank 0).

Default run (no ``--workload``): the headline workloads.

* ``value`` / ``ms_per_step`` / ``roofline`` / ``cpu_baseline`` / ``e2e``:
  the CIFAR-100-shaped soft training step (B = 2048, 46080 thermometer bits,
  two 128000-node layers, k = 6, 100 x 1280 group-sum head, tau = 100):
  thermometer encode, two LUT forwards, group-sum head with cross-entropy,
  layer-2 backward (table gradient + per-edge input-gradient terms), CSR
  reduction of the terms into layer 1's output gradient, layer-1 table
  gradient.
* ``hard``: the bit-packed evaluation of the CIFAR-10-shaped network
  (21504 bits, 64000 x 64000, k = 6, tables theta > 0) on 2^22 samples:
  table binarization, encode + pack, hard layer 1, hard layer 2 with the fused
  popcount head and argmax, with its own roofline, oracle baseline and
  end-to-end figure.
* ``extra``: the MNIST-shaped step at k = 6 and k = 2 and the
  CIFAR-10-shaped step (value, per-call split, roofline).

The two headline parts run one after the other, each over its own K timed
steps; the buffers of one are freed before the next is allocated.  L2 is
flushed between steps (a 512 MB write outside the timed events).  The timed
loops replay CUDA graphs captured once (no host work between launches); the
per-call split comes from eager steps with an event after every call.

  python bench.py [--gpus N] [--steps K] [--warmup W]          # headline
  python bench.py --workload mnist ...      # one workload (train + hard on its batch)
  python bench.py --impl reference ...      # the CPU oracle on the same workloads

Multi-GPU (torchrun, one process per GPU): every rank trains its own batch
and evaluates its own samples (weak scaling, no data-path collective); the
job's time is the max over ranks and ``value`` sums the samples of all
ranks.
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
FUSE = {"auto": None, "on": True, "off": False}
HEADLINE_TRAIN = "cifar100"
HEADLINE_HARD = "hard_cifar10"
EXTRAS = ("mnist", "mnist_k2", "cifar10")
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


def parse_args(argv=None):
    p = argparse.ArgumentParser()
    p.add_argument("--gpus", type=int, default=1)
    p.add_argument("--steps", type=int, default=30)
    p.add_argument("--warmup", type=int, default=5)
    p.add_argument("--impl", choices=["ours", "reference"], default="ours")
    p.add_argument("--workload", default=None, choices=sorted(synth.WORKLOADS),
                   help="one workload (training step plus the hard pass on its batch); "
                        "default: the headline workloads")
    p.add_argument("--extras", default=",".join(EXTRAS),
                   help="comma-separated training workloads reported under 'extra' in the headline run")
    p.add_argument("--no-extras", action="store_true")
    p.add_argument("--node", default="soft", choices=["soft", "st"],
                   help="LightLUT node form of the training step: soft, or straight-through hard")
    p.add_argument("--fuse-dy1", choices=["auto", "on", "off"], default="auto",
                   help="layer 1's backward sums layer 2's per-edge terms itself (no separate CSR reduction); "
                        "auto: when the terms are much larger than L2")
    p.add_argument("--through", choices=["auto", "on", "off"], default="auto",
                   help="layer 1 recomputes its output gradient through layer 2 (fan-in <= 3) instead of "
                        "reading layer 2's per-edge terms; auto: whenever layer 2's fan-in allows it")
    p.add_argument("--bytes1", choices=["auto", "on", "off"], default="auto",
                   help="layer 1 reads the encoder's wires as bytes: lookup forward and one-hot table "
                        "gradient (auto: whenever B % 4 == 0)")
    p.add_argument("--bits1", choices=["auto", "on", "off"], default="auto",
                   help="layer 1's binary wires kept at one bit per sample (wire bit rows) instead of a byte "
                        "(auto: on byte wires off the through route)")
    p.add_argument("--no-cpu-baseline", action="store_true")
    p.add_argument("--no-e2e", action="store_true")
    p.add_argument("--no-graph", action="store_true",
                   help="time eager launches instead of CUDA-graph replays of the step")
    p.add_argument("--profile", action="store_true",
                   help="plain timed loop only (for ncu launch lists)")
    p.add_argument("--batch", type=int, default=0,
                   help="override the workload's batch (smaller cases for ncu captures)")
    return p.parse_args(argv)


def peaks():
    """(HBM GB/s, SM max MHz, source) from the measured peaks file."""
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(path):
        with open(path) as f:
            m = json.load(f)
        return float(m["hbm_gbs"]), float(m.get("sm_max_mhz", 2070.0)), "measured"
    return 6800.0, 2070.0, "fallback"


def device_sms(device=None) -> int:
    """SM count of the device, read from the device."""
    return int(torch.cuda.get_device_properties(device if device is not None
                                                else torch.cuda.current_device()).multi_processor_count)


def issue_peak(sms: int, mhz: float) -> float:
    """Lane-operations per second at one warp instruction per clock and
    scheduler (128 lanes per SM)."""
    return sms * FP32_LANES_PER_SM * mhz * 1e6


# ------------------------------------------------------------- clocks --

class ClockSampler:
    """nvidia-smi samples of one GPU, taken only while a segment is open
    (start() .. stop()); summary() covers every segment so far."""

    def __init__(self, index: int, period_ms: int = 50):
        self.index, self.period = index, period_ms
        self.rows = []
        self.available = True
        self.proc = None

    def start(self):
        if not self.available:
            return
        try:
            fd, self.path = tempfile.mkstemp(suffix=".csv")
            os.close(fd)
            self.out = open(self.path, "w")
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--id={self.index}", f"--query-gpu={SMI_FIELDS}",
                 "--format=csv,noheader,nounits", "-lms", str(self.period)],
                stdout=self.out, stderr=subprocess.DEVNULL)
        except (OSError, FileNotFoundError):
            self.available = False
            self.proc = None
        time.sleep(0.1)   # let the first sample land inside the segment

    def stop(self) -> dict:
        seg = []
        if self.proc is not None:
            time.sleep(0.1)
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()
            self.out.close()
            with open(self.path) as f:
                for line in f:
                    parts = [p.strip() for p in line.split(",")]
                    if len(parts) >= 9:
                        seg.append(parts)
            os.unlink(self.path)
            self.proc = None
        self.rows.extend(seg)
        return self._summary(seg)

    def summary(self) -> dict:
        return self._summary(self.rows)

    def _summary(self, rows) -> dict:
        if not self.available:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": [], "samples": 0,
                    "note": "nvidia-smi unavailable"}
        sm, mx, pw, reasons = [], [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for parts in rows:
            try:
                sm.append(float(parts[1]))
                mx.append(float(parts[2]))
                pw.append(float(parts[3]))
            except ValueError:
                continue
            for name, val in zip(names, parts[5:9]):
                if val.lower().startswith("active"):
                    reasons.add(name)
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


def barrier(world: int):
    if world > 1:
        torch.distributed.barrier()


# ------------------------------------------------------ work per call --

def call_work_routed(wl, B):
    """Work of the calls of a routed training step: (algorithmic bytes, ops,
    bytes moved).  The routing calls count their HBM bytes (each slot's Kc
    candidate rows are gathered from the layer input, which stays in L2, so
    the gathered bytes are not HBM traffic) and one FMA per (candidate,
    sample); the LUT calls read the slot rows through the identity
    connectivity."""
    K, k, Kc = wl.K, wl.k, wl.Kc
    w1, w2 = wl.widths
    win, d, C = wl.w_in, wl.d, wl.classes
    s1, s2 = w1 * k, w2 * k
    f = 4
    W = (B + 31) // 32
    work = {
        # the encoder's wires are bytes in the routed step (layer 1 gathers them)
        "encode": (B * d + win * B, 0),
        "route1": (win * B + f * (s1 * B + 2 * s1 * Kc), Kc * s1 * B),
        "forward1": (f * (s1 * B + w1 * B + w1 * K + w1 * k), (2 * (K - 1) + k) * w1 * B),
        "route2": (f * (w1 * B + s2 * B + 2 * s2 * Kc), Kc * s2 * B),
        "forward2": (f * (s2 * B + w2 * B + w2 * K + w2 * k), (2 * (K - 1) + k) * w2 * B),
        "head": (f * (w2 * B + 2 * B * C + B), 0),
        "backward2": (f * (s2 * B + C * B + s2 * B + 2 * w2 * K + w2 * k), (4 * (K - 1) + K) * w2 * B),
        "route_bwd2": (f * (w1 * B + 2 * s2 * B + w1 * B + 3 * s2 * Kc), 2 * Kc * s2 * B),
        "backward1": (f * (s1 * B + w1 * B + s1 * B + 2 * w1 * K + w1 * k), (4 * (K - 1) + K) * w1 * B),
        "route_bwd1": (win * B + f * (s1 * B + 2 * s1 * Kc), Kc * s1 * B),
        "binarize": (f * (w1 * K + w2 * K) + 8 * (w1 + w2), 0),
        "pack": (B * d + f * win * W, 0),
        "hard1": (f * (win * W + w1 * W + w1 * k) + 8 * w1, (K - 1) * w1 * W),
        "hard2": (f * (w1 * W + w2 * k + B * C * 2 + B) + 8 * w2, (K - 1) * w2 * W),
    }
    return {n: (b, o, b) for n, (b, o) in work.items()}


def call_work(wl, B, fuse_dy1=False, through=False, bytes1=False, bits1=False):
    """Algorithmic work of each library call of one step on a batch of B:
    (algorithmic bytes, algorithmic ops, bytes the call moves).

    Ops follow the lerp-tree counts per (node, sample): forward 2(2^k-1)+k;
    backward with input gradient 4(2^k-1)+2^k; backward without it
    2(2^k-1)+2^k; hard layer 2^k-1 mux operations per (node, 32-sample word).
    Algorithmic bytes count each tensor the step must read or write once: the
    layer input X, the output gradient dY, the input gradient dX, the tables
    and their gradients, the connectivity and the CSR map.  The head's output
    gradient is one row per class (every node of a class has the same
    gradient), so dY is C x B, not w x B.  The per-edge input-gradient terms
    that the layer-2 backward writes and the CSR reduction reads are not
    algorithmic: they appear only in the bytes moved.

    With byte wires for layer 1 (``bytes1``) the encoder writes one byte per
    wire and layer 1's inputs are binary, so its corner weights are one-hot:
    the forward is a lookup (no arithmetic beyond the k-byte gather and one
    table read) and the table gradient one add per (node, sample); both
    calls are then bounded by their bytes.  With wire bit rows (``bits1``)
    each wire takes one bit per sample (32-bit words, 32 per 1024-sample
    block), written by the encoder and read by both layer-1 calls."""
    K, k = wl.K, wl.k
    w1, w2 = wl.widths
    win, d, C = wl.w_in, wl.d, wl.classes
    W = (B + 31) // 32
    f = 4
    terms = f * w2 * k * B
    csr2 = f * (w1 + 1 + w2 * k)
    work = {
        "encode": (B * d + f * win * B, 0, B * d + f * win * B),
        "forward1": (f * (win * B + w1 * B + w1 * K + w1 * k), (2 * (K - 1) + k) * w1 * B, None),
        "forward2": (f * (w1 * B + w2 * B + w2 * K + w2 * k), (2 * (K - 1) + k) * w2 * B, None),
        # reads Y2 and the labels; writes the logits and one gradient row per class
        "head": (f * (w2 * B + 2 * B * C + B), 0, None),
        # §8(a) a4 with dX for layer 2 is backward2 + csr2: X = Y1, dY rows,
        # the table and its gradient, the connectivity (here), the CSR map and
        # dX = dY1 (the reduction); both calls carry the per-edge terms
        "backward2": (f * (w1 * B + C * B + 2 * w2 * K + w2 * k), (4 * (K - 1) + K) * w2 * B,
                      f * (w1 * B + C * B + 2 * w2 * K + w2 * k) + terms),
        "csr2": (f * w1 * B + csr2, 0, f * w1 * B + csr2 + terms),
        "backward1": (f * (win * B + w1 * B + 2 * w1 * K + w1 * k), (2 * (K - 1) + K) * w1 * B, None),
        "binarize": (f * (w1 * K + w2 * K) + 8 * (w1 + w2), 0, None),
        "pack": (B * d + f * win * W, 0, None),
        "hard1": (f * (win * W + w1 * W + w1 * k) + 8 * w1, (K - 1) * w1 * W, None),
        "hard2": (f * (w1 * W + w2 * k + B * C * 2 + B) + 8 * w2, (K - 1) * w2 * W, None),
    }
    xb1 = 1 if bytes1 else f   # bytes per layer-1 input value
    dth1_ops = w1 * B if bytes1 else (2 * (K - 1) + K) * w1 * B   # layer-1 table gradient
    if bytes1:
        # byte rows: the encoder writes one byte per wire, the layer-1
        # forward gathers bytes and reads one table entry per output
        work["encode"] = (B * d + win * B, 0, B * d + win * B)
        work["forward1"] = (win * B + f * (w1 * B + w1 * K + w1 * k), 0, None)
        work["backward1"] = (win * B + f * (w1 * B + 2 * w1 * K + w1 * k), dth1_ops, None)
    if bits1:
        xw1 = 4 * win * (32 * ((B + 1023) // 1024))   # the wire bit rows
        work["encode"] = (B * d + xw1, 0, B * d + xw1)
        work["forward1"] = (xw1 + f * (w1 * B + w1 * K + w1 * k), 0, None)
        work["backward1"] = (xw1 + f * (w1 * B + 2 * w1 * K + w1 * k), dth1_ops, None)
    if through:
        # layer 2: table gradient only; layer 1: its table gradient with its
        # output gradient recomputed through layer 2 (the consumers' other
        # inputs from Y1, the per-class rows, layer 2's tables, connectivity
        # and CSR map), so the a4 row's input-gradient work for layer 2 moves
        # to backward1 and nothing per edge is stored
        work["backward2"] = (f * (w1 * B + C * B + 2 * w2 * K + w2 * k), (2 * (K - 1) + K) * w2 * B, None)
        work["backward1"] = (xb1 * win * B + f * (w1 * B + C * B + 2 * w1 * K + w1 * k + w2 * K + w2 * k) + csr2,
                             dth1_ops + 2 * (K - 1) * w2 * B, None)
        del work["csr2"]
        return {n: (b, o, b if m is None else m) for n, (b, o, m) in work.items()}
    if fuse_dy1:
        # layer 1 sums layer 2's per-edge terms through the CSR map itself
        xin = xw1 if bits1 else xb1 * win * B
        work["backward1"] = (xin + f * (w1 * B + 2 * w1 * K + w1 * k) + csr2, dth1_ops,
                             xin + f * (2 * w1 * K + w1 * k) + csr2 + terms)
        del work["csr2"]
    return {n: (b, o, b if m is None else m) for n, (b, o, m) in work.items()}


# DRAM traffic per launch of a roofline kernel, dram__bytes_read.sum +
# dram__bytes_write.sum from one ncu capture, keyed by workload and call.
# Valid only for the kernel source it was taken on: the SHA-256 of the
# source file's code (comments and blank space removed) is recorded, and any
# later change of the code reports null.
TRAFFIC = {
    ("mnist", "backward2"): {
        "bytes": 59560448 + 144350720, "source": "lut_soft.cu",
        "sha256": "78edac247d6c64dc0042c15287b5174dfc03ecac6e7945ec4beb26e9e6cc6800",
        "note": "ncu capture of this workload (one-pass DRAM metrics)"},
    ("cifar10", "forward2"): {
        "bytes": 1162980096 + 245190144, "source": "lut_soft.cu",
        "sha256": "78edac247d6c64dc0042c15287b5174dfc03ecac6e7945ec4beb26e9e6cc6800",
        "note": "ncu capture of this workload (one-pass DRAM metrics)"},
    ("cifar10", "backward2"): {
        "bytes": 1344603136 + 1542144768, "source": "lut_soft.cu",
        "sha256": "78edac247d6c64dc0042c15287b5174dfc03ecac6e7945ec4beb26e9e6cc6800",
        "note": "ncu capture of this workload (one-pass DRAM metrics)"},
    ("cifar100", "forward2"): {
        "bytes": 5876089344 + 1032741376, "source": "lut_soft.cu",
        "sha256": "78edac247d6c64dc0042c15287b5174dfc03ecac6e7945ec4beb26e9e6cc6800",
        "note": "ncu capture of this workload (one-pass DRAM metrics)"},
    ("cifar100", "backward2"): {
        "bytes": 6068320768 + 6277417984, "source": "lut_soft.cu",
        "sha256": "78edac247d6c64dc0042c15287b5174dfc03ecac6e7945ec4beb26e9e6cc6800",
        "note": "ncu capture of this workload (one-pass DRAM metrics)"},
    ("cifar10", "forward1"): {
        "bytes": 20694272 + 196729088, "source": "lut_bytes.cu",
        "sha256": "88cd7e78b309d49ee5835ba21aeb26fbdf1a8e144188cac4f9338e562f6c3f57",
        "note": "ncu capture of this workload (one-pass DRAM metrics)"},
    ("cifar10", "backward1"): {
        "bytes": 1594112256 + 4992000, "source": "lut_through.cu",
        "sha256": "ad4bbdb6659e473eed215cff59a03a8b3529059b4611af7795cf503b7e580392",
        "note": "ncu capture of this workload (one-pass DRAM metrics)"},
    ("cifar100", "forward1"): {
        "bytes": 50327040 + 984133120, "source": "lut_bytes.cu",
        "sha256": "88cd7e78b309d49ee5835ba21aeb26fbdf1a8e144188cac4f9338e562f6c3f57",
        "note": "ncu capture of this workload (one-pass DRAM metrics)"},
    ("cifar100", "backward1"): {
        "bytes": 6341038592 + 8354816, "source": "lut_through.cu",
        "sha256": "ad4bbdb6659e473eed215cff59a03a8b3529059b4611af7795cf503b7e580392",
        "note": "ncu capture of this workload (one-pass DRAM metrics)"},
    ("cifar10", "encode"): {
        "bytes": 3160576 + 0, "source": "encode.cu",
        "sha256": "e6c29181c8e57f1b0f92ecd6dfdad87e8d79378c78599c3d42e80904a0b689a6",
        "note": "ncu capture of this workload (one-pass DRAM metrics)"},
    ("cifar100", "encode"): {
        "bytes": 6312448 + 0, "source": "encode.cu",
        "sha256": "e6c29181c8e57f1b0f92ecd6dfdad87e8d79378c78599c3d42e80904a0b689a6",
        "note": "ncu capture of this workload (one-pass DRAM metrics)"},
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
    "forward2": "lut_forward_staged_kernel<k>", "head": "head_group_sum + head_softmax (2 kernels)",
    "backward2": "lut_backward_node_kernel<k, dx, dY rows>",
    "backward1": "lut_backward_theta_kernel<k>", "csr2": "csr_reduce_kernel",
    "binarize": "binarize_kernel (x2)", "pack": "pack_bits_kernel", "hard1": "hard_layer_staged_kernel<k>",
    "hard2": "hard_head_staged_kernel<k> + argmax_kernel",
    "route1": "route_forward_vec_kernel<KC>", "route2": "route_forward_vec_kernel<KC>",
    "route_bwd2": "route_dr_kernel + route_dx_kernel", "route_bwd1": "route_dr_kernel<KC> (byte rows)",
}
# calls that launch more than one kernel: not a single-kernel roofline
MULTI_KERNEL_CALLS = ("head", "binarize", "hard2", "route_bwd2")


def route_of_step(st) -> dict:
    """How the step runs layer 1: its input wires and where its output
    gradient comes from."""
    if getattr(st, "through", False):
        grad = "recomputed through layer 2 (fan-in <= 3)"
    elif getattr(st, "fuse_dy1", False):
        grad = "layer 2's per-edge terms summed in the layer-1 kernel"
    else:
        grad = "CSR reduction of layer 2's per-edge terms"
    wires = ("bytes: lookup forward, one-hot table gradient" if getattr(st, "bytes1", False)
             else "fp32: lerp-tree forward, multilinear table gradient")
    if getattr(st, "bits1", False):
        wires = "bits (one per sample): lookup forward, one-hot table gradient"
    return {"layer1_wires": wires, "layer1_output_gradient": grad}


def kernels_of_step(st) -> dict:
    """The kernel behind each call of a training step, by its route: byte
    wires for layer 1 or fp32, the fused, through or CSR route for layer 1's
    output gradient."""
    names = dict(KERNEL_OF_CALL)
    if getattr(st, "bits1", False):
        names["encode"] = "encode_bitrows_kernel"
        names["forward1"] = "lut_forward_bits_kernel<k> (lookup)"
    elif getattr(st, "bytes1", False):
        names["encode"] = "encode_soft_vec_kernel<uint8_t>"
        names["forward1"] = "lut_forward_u8_kernel<k> (lookup)"
    through, fused = getattr(st, "through", False), getattr(st, "fuse_dy1", False)
    if through:
        names["backward2"] = "lut_backward_theta_kernel<k> (dtheta only, class rows)"
        names["backward1"] = "lut_theta_through_kernel<k, ku, " + ("uint8_t>" if st.bytes1 else "float>")
    elif getattr(st, "bytes1", False):
        src = "bit rows" if getattr(st, "bits1", False) else "byte rows"
        names["backward1"] = (f"lut_theta_bytes_kernel<k, terms, {src}> (one-hot)" if fused
                              else f"lut_theta_bytes_kernel<k, dY rows, {src}> (one-hot)")
    elif fused:
        names["backward1"] = "lut_backward_node_kernel<k, 0, terms>"
    return names


def roofline_of(call, work, per_call_ms, sms, clocks, workload, hbm, sm_max, peak_kind, kernels=None):
    """Roofline object of one single-kernel call: the bound (HBM bytes or
    issue-rate lane-operations, whichever takes longer at peak), achieved
    rate, peak, fraction (also at the median SM clock sampled during the
    timed region) and the ncu DRAM traffic per launch."""
    byts, ops, moved = work[call]
    t_s = per_call_ms[call] * 1e-3
    alu_peak = issue_peak(sms, sm_max)
    t_hbm, t_alu = byts / (hbm * 1e9), ops / alu_peak
    if t_alu >= t_hbm:
        unit = ("Tops/s (integer mux lane-ops against the issue rate)" if call.startswith("hard")
                else "Tops/s (fp32 pipe lane-ops)")
        roof = {"bound": "alu", "achieved": ops / t_s / 1e12, "peak": alu_peak / 1e12, "unit": unit}
        med = clocks.get("sm_mhz")
        if med:
            roof["frac_at_sampled_clock"] = ops / t_s / issue_peak(sms, med)
    else:
        roof = {"bound": "hbm", "achieved": byts / t_s / 1e9, "peak": hbm, "unit": "GB/s"}
    roof["frac"] = roof["achieved"] / roof["peak"]
    traffic, traffic_note = kernel_traffic(workload, call)
    roof.update({"traffic": traffic, "traffic_source": traffic_note,
                 "traffic_over_algorithmic": (traffic / byts) if traffic else None,
                 "kernel": (kernels or KERNEL_OF_CALL)[call], "call": call,
                 "ms_per_launch": per_call_ms[call], "algorithmic_bytes": byts, "bytes_moved": moved,
                 "algorithmic_ops": ops,
                 "peak_source": f"{peak_kind} HBM copy ({hbm:.1f} GB/s); {sms} SMs (read from the device) x "
                                f"{FP32_LANES_PER_SM} lanes x {sm_max:.0f} MHz (alu: one issue per lane and clock)"})
    return roof


def calls_table(work, per_call_ms, hbm, workload=None, kernels=None):
    out = {}
    for n, t in per_call_ms.items():
        b_, o_, m_ = work[n]
        e = {"ms": round(t, 5), "alg_GB/s": round(b_ / (t * 1e-3) / 1e9, 1),
             "frac_hbm": round(b_ / (t * 1e-3) / 1e9 / hbm, 3),
             "Tops/s": round(o_ / (t * 1e-3) / 1e12, 2) if o_ else None}
        if m_ != b_:
            e["moved_GB/s"] = round(m_ / (t * 1e-3) / 1e9, 1)
        traffic, _ = kernel_traffic(workload, n) if workload else (None, None)
        if traffic:
            # DRAM bytes per launch from ncu against the algorithmic bytes,
            # and the DRAM rate they imply at the event-timed duration
            e["traffic_over_algorithmic"] = round(traffic / b_, 2)
            e["dram_GB/s"] = round(traffic / (t * 1e-3) / 1e9, 1)
        if kernels and n in kernels:
            e["kernel"] = kernels[n]
        out[n] = e
    return out


def step_bytes(wl, B):
    """Algorithmic bytes of one training step (thermometer encode, two LUT
    forwards, head + cross-entropy, layer-2 backward with the input gradient,
    layer-1 backward without it), each tensor moved once, whatever calls the
    step is split into.  "survey": every node has its own output-gradient row
    (the head writes dY as w x B and the layer-2 backward reads it);
    "design": the head writes one gradient row per class (C x B), which every
    node of the class reads."""
    K, k = wl.K, wl.k
    w1, w2 = wl.widths
    win, d, C = wl.w_in, wl.d, wl.classes
    f = 4
    enc = B * d + f * win * B
    fwd = f * (win * B + w1 * B + w1 * K + w1 * k) + f * (w1 * B + w2 * B + w2 * K + w2 * k)
    csr2, csr1 = f * (w1 + 1 + w2 * k), f * (win + 1 + w1 * k)
    bwd1 = f * (win * B + w1 * B + 2 * w1 * K) + csr1
    survey = enc + fwd + f * (2 * w2 * B) + f * (w1 * B + w2 * B + w1 * B + 2 * w2 * K) + csr2 + bwd1
    design = enc + fwd + f * (w2 * B + 2 * B * C + B) + f * (w1 * B + C * B + w1 * B + 2 * w2 * K) + csr2 + bwd1
    return {"survey": survey, "design": design}


def step_hbm_fraction(wl, B, work, names, ms_step, hbm):
    """The step's algorithmic bytes over the step time, against the HBM
    peak, with the bytes the calls actually move (per-edge terms included)."""
    sb = step_bytes(wl, B)
    moved = sum(work[n][2] for n in names if n in work)
    t = ms_step * 1e-3
    return {"algorithmic_bytes": sb["design"], "alg_GB/s": sb["design"] / t / 1e9,
            "frac_hbm": sb["design"] / t / 1e9 / hbm,
            "algorithmic_bytes_survey": sb["survey"], "frac_hbm_survey": sb["survey"] / t / 1e9 / hbm,
            "bytes_moved": moved, "moved_over_algorithmic": moved / sb["design"],
            "note": "design bytes: per-class output-gradient rows (C x B); survey bytes: one row per node (w x B)"}


# --------------------------------------------------------------- ours --

def dist_env():
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return world, rank, local


def with_batch(wl, batch):
    if not batch:
        return wl
    return synth.Workload(wl.name, batch, wl.d, wl.classes, wl.sigma, wl.thresholds, wl.widths, wl.k, wl.tau,
                          wl.Kc)


class Timer:
    """Timed loops and eager per-call splits over one step function, with L2
    flushed before every step and CUDA events on the launching stream."""

    def __init__(self, flush, stream, clock, world):
        self.flush, self.stream, self.clock, self.world = flush, stream, clock, world

    def timed(self, replay, K):
        """ms of each of K steps (events around each replay) and the clocks
        sampled during the loop."""
        barrier(self.world)
        torch.cuda.synchronize()
        self.clock.start()
        wall0 = time.perf_counter()
        evs = []
        for _ in range(K):
            self.flush.fill_(1)
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record(self.stream)
            replay()
            e1.record(self.stream)
            evs.append((e0, e1))
        torch.cuda.synchronize()
        wall = time.perf_counter() - wall0
        barrier(self.world)
        clocks = self.clock.stop()
        return [a.elapsed_time(b) for a, b in evs], clocks, wall

    def eager_split(self, step, n):
        """n eager steps with an event after every library call: mean ms per
        call and per step.  Each step is queued behind a short bounded sleep
        kernel (about 1 ms), so the host has enqueued the whole step before
        the GPU reaches it and the events time the kernels, not the host's
        launch path."""
        marks = []
        for _ in range(n):
            self.flush.fill_(1)
            torch.cuda._sleep(2_000_000)
            lst = []
            marks.append(lst)

            def mark(name, lst=lst):
                ev = torch.cuda.Event(enable_timing=True)
                ev.record(self.stream)
                lst.append((name, ev))
            mark("start")
            step(mark)
        torch.cuda.synchronize()
        calls, totals = {}, []
        for lst in marks:
            prev = lst[0][1]
            tot = 0.0
            for name, ev in lst[1:]:
                dt = prev.elapsed_time(ev)
                prev = ev
                calls.setdefault(name, []).append(dt)
                tot += dt
            totals.append(tot)
        return {n: float(np.mean(v)) for n, v in calls.items()}, float(np.mean(totals))

    def event_floor(self, n=30):
        """ms the eager split reports for a near-empty kernel (the issue
        probe with one iteration: one block of 1024 threads per SM) placed
        where a step's first call sits: the launch and event overhead that
        every entry of the split carries."""
        import paper_2602_07400_gb300 as bl
        if not hasattr(self, "_floor_sink"):
            self._floor_sink = torch.empty(bl.bitlogic_issue_probe_threads(), dtype=torch.int32, device="cuda")

        def step(mark):
            bl.bitlogic_issue_probe("ffma", 1, self._floor_sink)
            mark("empty")
        per_call, _ = self.eager_split(step, n)
        return per_call["empty"]


def build_train(wl, rank, node="soft", fuse_dy1=None, through=None, bytes1=None, bits1=None):
    from paper_2602_07400_gb300.pipeline import Network, RoutedNetwork, RoutedTrainStep, TrainStep
    B = wl.batch
    if wl.Kc:
        rnet = RoutedNetwork(*synth.routed_network(wl, seed=0), wl.w_in)
        st = RoutedTrainStep(rnet, B, wl.d, wl.thresholds, wl.classes, wl.tau, node=node)
        net = rnet
    else:
        conn1, th1, conn2, th2 = synth.network(wl, seed=0)
        net = Network(conn1, th1, conn2, th2, wl.w_in)
        st = TrainStep(net, B, wl.d, wl.thresholds, wl.classes, wl.tau, node=node, fuse_dy1=fuse_dy1,
                       through=through, bytes1=bytes1, bits1=bits1)
    x, lab = synth.blob_batch(B, wl.d, wl.classes, wl.sigma, seed=1000 + rank)
    st.load(x.cuda(), lab.cuda())
    return net, st


def measure_train(wl, st, args, timer, hbm, sm_max, peak_kind, sms, world, detail=True):
    """Timed training steps of ``st`` (graph replays unless --no-graph), the
    per-call split and the roofline of the dominant single-kernel call."""
    import paper_2602_07400_gb300 as bl
    B, K = wl.batch, args.steps
    for _ in range(args.warmup):
        timer.flush.fill_(1)
        st.run()
    torch.cuda.synchronize()
    use_graph = not (args.no_graph or args.profile)
    if use_graph:
        g = st.capture()
        for _ in range(3):
            timer.flush.fill_(1)
            g.replay()
        torch.cuda.synchronize()
        ms, clocks, wall = timer.timed(g.replay, K)
    else:
        ms, clocks, wall = timer.timed(st.run, K)
    assert bl.bitlogic_device_error() == 0
    tot = max_over_ranks([sum(ms)], "cuda")[0]
    per_call, eager_step = timer.eager_split(lambda mark: st.run(mark=mark), max(3, min(K, 30)))
    work = call_work_routed(wl, B) if wl.Kc else call_work(wl, B, fuse_dy1=st.fuse_dy1,
                                                              through=getattr(st, "through", False),
                                                              bytes1=getattr(st, "bytes1", False),
                                                              bits1=getattr(st, "bits1", False))
    single = {n: t for n, t in per_call.items() if n not in MULTI_KERNEL_CALLS}
    dom = max(single, key=single.get)
    res = {
        "value": job_rate(world, B, K, tot), "unit": "samples/s", "ms_per_step": tot / K,
        "eager_ms_per_step": eager_step,
        "roofline": roofline_of(dom, work, per_call, sms, clocks, wl.name, hbm, sm_max, peak_kind,
                                kernels=None if wl.Kc else kernels_of_step(st)),
        "calls": calls_table(work, per_call, hbm, wl.name, kernels=None if wl.Kc else kernels_of_step(st)),
        "calls_event_floor_ms": timer.event_floor(),
        "route": None if wl.Kc else route_of_step(st),
        "step_hbm": step_hbm_fraction(wl, B, work, per_call.keys(), tot / K, hbm) if not wl.Kc else None,
        "gpu_launches": K * st.kernels_per_run,
        "clocks": clocks, "wall_s_timed_loop": wall,
        "timing": ("CUDA-graph replays of the training step (fwd+bwd), CUDA events around each replay; "
                   "per-call split from eager steps queued behind a 1 ms sleep, an event after every call"
                   if use_graph else "eager launches, CUDA events around each step"),
    }
    if detail:
        res["roofline_by_call"] = {n: {k_: v for k_, v in roofline_of(n, work, per_call, sms, clocks, wl.name,
                                                                      hbm, sm_max, peak_kind).items()
                                       if k_ in ("bound", "frac", "frac_at_sampled_clock", "achieved", "unit")}
                                   for n in single}
    return res


def build_hard(wl, net, rank, x_dev=None):
    from paper_2602_07400_gb300.pipeline import HardInfer
    hi = HardInfer(net, wl.batch, wl.d, wl.thresholds, wl.classes)
    if x_dev is not None:
        hi.x = x_dev                 # evaluate the training batch
    else:
        x, _ = synth.blob_batch(wl.batch, wl.d, wl.classes, wl.sigma, seed=1000 + rank, device="cuda")
        hi.x.copy_(x)
        del x
    return hi


def measure_hard(wl, hi, args, timer, hbm, sm_max, peak_kind, sms, world):
    """Timed hard passes (binarize + pack + 2 layers + popcount head + argmax)."""
    import paper_2602_07400_gb300 as bl
    N, K = wl.batch, args.steps
    for _ in range(max(1, args.warmup)):
        timer.flush.fill_(1)
        hi.binarize()
        hi.run()
    torch.cuda.synchronize()
    use_graph = not (args.no_graph or args.profile)
    if use_graph:
        g = hi.capture(binarize=True)
        for _ in range(2):
            timer.flush.fill_(1)
            g.replay()
        torch.cuda.synchronize()
        ms, clocks, wall = timer.timed(g.replay, K)
    else:
        ms, clocks, wall = timer.timed(lambda: (hi.binarize(), hi.run()), K)
    assert bl.bitlogic_device_error() == 0
    tot = max_over_ranks([sum(ms)], "cuda")[0]

    def step(mark):
        hi.binarize(mark=mark)
        hi.run(mark=mark)
    n_split = max(3, min(K, 100 if N <= (1 << 16) else 10))
    per_call, eager_step = timer.eager_split(step, n_split)
    work = call_work(wl, N)
    per_call_w = {n: t for n, t in per_call.items()}
    res = {
        "value": job_rate(world, N, K, tot) / 1e6, "unit": "MSamples/s", "ms_per_batch": tot / K,
        "batch": N, "eager_ms_per_batch": eager_step,
        "includes": "binarize + encode/pack + 2 hard layers + popcount head + argmax",
        "calls": calls_table(work, per_call_w, hbm, wl.name),
        "gpu_launches": K * (hi.kernels_per_binarize + hi.kernels_per_run),
        "clocks": clocks, "wall_s_timed_loop": wall,
    }
    roof = roofline_of("hard1", work, per_call_w, sms, clocks, wl.name, hbm, sm_max, peak_kind)
    res["roofline"] = roof
    # layer 2 with the fused head: its mux tree against the same peak (the
    # call also runs the argmax kernel, a few hundred microseconds at 2^22)
    r2 = roofline_of("hard2", work, per_call_w, sms, clocks, wl.name, hbm, sm_max, peak_kind)
    res["roofline_hard2"] = {k_: r2[k_] for k_ in ("bound", "achieved", "peak", "unit", "frac", "ms_per_launch")
                             if k_ in r2}
    return res


def run_e2e_train(st, wl, K, world, rank, use_graph=True):
    """The training metric end to end through the public API: every step
    copies its batch (raw uint8 samples and labels) from pinned host memory
    and reads the loss back.  With graphs, ``pipeline.Prefetcher`` overlaps
    the copy of the next batch with the current step (two input buffers, a
    copy stream); without, the copy, the step and the read-back run in
    sequence."""
    from paper_2602_07400_gb300.pipeline import Prefetcher
    B = wl.batch
    x_host, lab_host = synth.blob_batch(B, wl.d, wl.classes, wl.sigma, seed=2000 + rank)
    x_host, lab_host = x_host.pin_memory(), lab_host.pin_memory()
    loss_host = torch.empty(1, dtype=torch.float32).pin_memory()

    def eager():
        st.load(x_host, lab_host, non_blocking=True)
        st.run()
        loss_host.copy_(st.loss, non_blocking=True)
    pf = Prefetcher(st, ("x", "labels"), "loss") if use_graph else None
    ms = _e2e_loop(pf, {"x": x_host, "labels": lab_host}, loss_host, eager, K)
    return {"value": job_rate(world, B, K, ms), "unit": "samples/s",
            "h2d_bytes_per_step": x_host.numel() + 4 * lab_host.numel(),
            "d2h_bytes_per_step": 4, "overlap": bool(use_graph)}


def run_e2e_hard(hi, wl, K, world, rank, use_graph=True):
    """The hard metric end to end: every batch of raw samples is copied from
    pinned host memory and the predictions are read back.  For the large
    batches the host copy of the samples is taken from the device-generated
    batch (drawing 2^22 x 3072 pixels on the host would take minutes)."""
    from paper_2602_07400_gb300.pipeline import Prefetcher
    N = wl.batch
    if N > (1 << 16):
        x_host = torch.empty(N, wl.d, dtype=torch.uint8).pin_memory()
        x_host.copy_(hi.x)
    else:
        x_host, _ = synth.blob_batch(N, wl.d, wl.classes, wl.sigma, seed=2000 + rank)
        x_host = x_host.pin_memory()
    pred_host = torch.empty(N, dtype=torch.int32).pin_memory()

    def eager():
        hi.x.copy_(x_host, non_blocking=True)
        hi.binarize()
        hi.run()
        pred_host.copy_(hi.pred, non_blocking=True)
    pf = Prefetcher(hi, ("x",), "pred", capture=lambda: hi.capture(binarize=True)) if use_graph else None
    ms = _e2e_loop(pf, {"x": x_host}, pred_host, eager, K)
    del pf
    return {"value": job_rate(world, N, K, ms) / 1e6, "unit": "MSamples/s",
            "h2d_bytes_per_step": x_host.numel(), "d2h_bytes_per_step": 4 * N, "overlap": bool(use_graph)}


def _e2e_loop(pf, host, res, eager, K):
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


def free_cuda():
    import gc
    gc.collect()
    torch.cuda.synchronize()
    torch.cuda.empty_cache()


def config_of(wl, world, node="soft"):
    return {"workload": wl.name, "batch_per_gpu": wl.batch, "d": wl.d, "thresholds": list(wl.thresholds),
            "widths": list(wl.widths), "k": wl.k, "classes": wl.classes, "tau": wl.tau,
            "routing": f"learnable, {wl.Kc} candidates per slot" if wl.Kc else "fixed (random-unique)",
            "node": "LightLUT " + ("soft" if node == "soft" else "straight-through hard"),
            "l2": "flushed between steps (512 MB write outside the timed events)",
            "parallelism": f"dp{world} (independent batches, no collective)"}


def base_line(world, K, W):
    return {"metric": METRIC, "n_gpus": world, "steps": K, "warmup": W, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f32",
            "data": "synthetic (seeded class-conditional Gaussian blobs, MNIST/CIFAR shapes; random-init tables)"}


def run_headline(args):
    """The default run: CIFAR-100-shaped training (value), 2^22-sample hard
    pass of the CIFAR-10-shaped network (hard), extra training workloads."""
    import paper_2602_07400_gb300 as bl
    world, rank, local = dist_env()
    hbm, sm_max, peak_kind = peaks()
    sms = device_sms(local)
    flush = torch.empty(512 << 20, dtype=torch.uint8, device="cuda")
    stream = torch.cuda.current_stream()
    clock = ClockSampler(local)
    timer = Timer(flush, stream, clock, world)
    use_graph = not (args.no_graph or args.profile)
    K = args.steps

    # -- headline training workload
    wl = with_batch(synth.WORKLOADS[HEADLINE_TRAIN], args.batch)
    net, st = build_train(wl, rank, args.node, FUSE[args.fuse_dy1], FUSE[args.through], FUSE[args.bytes1], FUSE[args.bits1])
    train = measure_train(wl, st, args, timer, hbm, sm_max, peak_kind, sms, world)
    upd = time_update(st, max(3, min(K, 20)))
    n_par = int(net.theta1.numel() + net.theta2.numel())
    optimizer = {"ms_per_update": upd, "kernel": "adamw_vec_kernel (x2)", "algorithmic_bytes": 28 * n_par,
                 "GB/s": 28 * n_par / (upd * 1e-3) / 1e9,
                 "settings": "AdamW beta (0.9, 0.999), eps 1e-8, lr 0.01, wd 0"}
    dp = time_dp_exchange(st, world) if world > 1 else None
    e2e = None if (args.no_e2e or args.profile) else run_e2e_train(st, wl, K, world, rank, use_graph)
    del st, net
    free_cuda()

    # -- headline hard workload (its own network and 2^22 samples)
    wh = synth.WORKLOADS[HEADLINE_HARD]
    if args.batch:
        wh = with_batch(wh, max(32, args.batch))
    from paper_2602_07400_gb300.pipeline import Network
    conn1, th1, conn2, th2 = synth.network(wh, seed=0)
    hnet = Network(conn1, th1, conn2, th2, wh.w_in)
    hi = build_hard(wh, hnet, rank)
    hard = measure_hard(wh, hi, args, timer, hbm, sm_max, peak_kind, sms, world)
    if not args.profile:
        rates = measure_pipe_rates(sms)
        hard["roofline"] = hard_roofline(hard["roofline"], rates, sms, hard["clocks"])
        r2 = hard_roofline(hard["roofline_hard2"], rates, sms, hard["clocks"])
        hard["roofline_hard2"] = {k_: r2[k_] for k_ in ("bound", "achieved", "peak", "unit", "frac",
                                                       "frac_issue_rate", "ms_per_launch")}
    if not (args.no_e2e or args.profile):
        hard["e2e"] = run_e2e_hard(hi, wh, K, world, rank, use_graph)
    hard["config"] = config_of(wh, world)
    del hi, hnet
    free_cuda()

    # -- extra training workloads: value, split and roofline each
    extra = {}
    names = [] if (args.no_extras or args.profile) else [n for n in args.extras.split(",") if n]
    for name in names:
        we = synth.WORKLOADS[name]
        enet, est = build_train(we, rank, args.node, FUSE[args.fuse_dy1], FUSE[args.through], FUSE[args.bytes1], FUSE[args.bits1])
        r = measure_train(we, est, args, timer, hbm, sm_max, peak_kind, sms, world, detail=False)
        r["config"] = {k_: v for k_, v in config_of(we, world, args.node).items()
                       if k_ in ("workload", "batch_per_gpu", "widths", "k", "classes", "tau")}
        extra[name] = r
        del est, enet
        free_cuda()

    if rank != 0:
        return None
    out = base_line(world, K, args.warmup)
    out.update({
        "value": train["value"], "unit": "samples/s", "ms_per_step": train["ms_per_step"],
        "config": config_of(wl, world, args.node),
        "roofline": train["roofline"],
        "gpu_launches": train["gpu_launches"],
        "clocks": train["clocks"],
        "timing": train["timing"],
        "eager_ms_per_step": train["eager_ms_per_step"],
        "calls": train["calls"],
        "calls_event_floor_ms": train["calls_event_floor_ms"],
        "route": train["route"],
        "roofline_by_call": train["roofline_by_call"],
        "step_hbm": train["step_hbm"],
        "wall_s_timed_loop": train["wall_s_timed_loop"],
        "optimizer": optimizer,
        "hard": hard,
        "extra": extra,
        "clocks_all_timed_loops": clock.summary(),
        "gpu_launches_all_timed_loops": train["gpu_launches"] + hard["gpu_launches"] +
        sum(v["gpu_launches"] for v in extra.values()),
    })
    if dp:
        out["dp_exchange"] = dp
    if e2e:
        out["e2e"] = e2e
    if not args.profile:
        out["fit"] = time_quantile_fit(wl, flush)
        out["pipe_rates"] = rates
    return out


def run_single(args):
    """One workload: its training step and the hard pass on the same batch
    (or the hard pass alone for the hard workloads)."""
    import paper_2602_07400_gb300 as bl
    world, rank, local = dist_env()
    hbm, sm_max, peak_kind = peaks()
    sms = device_sms(local)
    wl = with_batch(synth.WORKLOADS[args.workload], args.batch)
    hard_only = wl.name.startswith("hard_")
    flush = torch.empty(512 << 20, dtype=torch.uint8, device="cuda")
    stream = torch.cuda.current_stream()
    clock = ClockSampler(local)
    timer = Timer(flush, stream, clock, world)
    use_graph = not (args.no_graph or args.profile)
    K = args.steps
    train = None
    if hard_only:
        from paper_2602_07400_gb300.pipeline import Network
        net = Network(*synth.network(wl, seed=0), wl.w_in)
        hi = build_hard(wl, net, rank)
    else:
        rnet, st = build_train(wl, rank, args.node, FUSE[args.fuse_dy1], FUSE[args.through], FUSE[args.bytes1], FUSE[args.bits1])
        net = rnet.snap() if wl.Kc else rnet   # the hard pass evaluates the discretized network
        train = measure_train(wl, st, args, timer, hbm, sm_max, peak_kind, sms, world)
        hi = build_hard(wl, net, rank, x_dev=st.x)
    hard = measure_hard(wl, hi, args, timer, hbm, sm_max, peak_kind, sms, world)
    rates = None
    if not args.profile:
        rates = measure_pipe_rates(sms)
        hard["roofline"] = hard_roofline(hard["roofline"], rates, sms, hard["clocks"])
        r2 = hard_roofline(hard["roofline_hard2"], rates, sms, hard["clocks"])
        hard["roofline_hard2"] = {k_: r2[k_] for k_ in ("bound", "achieved", "peak", "unit", "frac",
                                                       "frac_issue_rate", "ms_per_launch")}
    e2e_train = e2e_hard = None
    if not (args.no_e2e or args.profile):
        if train is not None:
            e2e_train = run_e2e_train(st, wl, K, world, rank, use_graph)
        e2e_hard = run_e2e_hard(hi, wl, K, world, rank, use_graph)
    optimizer = None
    if train is not None and not args.profile:
        upd = time_update(st, max(3, min(K, 50)))
        n_par = int(st.net.theta1.numel() + st.net.theta2.numel())
        if wl.Kc:
            n_par += int(st.net.r1.numel() + st.net.r2.numel())
        optimizer = {"ms_per_update": upd, "kernel": f"adamw_vec_kernel (x{4 if wl.Kc else 2})",
                     "algorithmic_bytes": 28 * n_par, "GB/s": 28 * n_par / (upd * 1e-3) / 1e9,
                     "settings": "AdamW beta (0.9, 0.999), eps 1e-8, lr 0.01, wd 0"}
    dp = time_dp_exchange(st, world) if (train is not None and world > 1 and not args.profile) else None
    if rank != 0:
        return None
    out = base_line(world, K, args.warmup)
    main = train if train is not None else hard
    out.update({
        "value": train["value"] if train else hard["value"],
        "unit": "samples/s" if train else "MSamples/s",
        "ms_per_step": train["ms_per_step"] if train else hard["ms_per_batch"],
        "config": config_of(wl, world, args.node),
        "roofline": main["roofline"],
        "gpu_launches": main["gpu_launches"],
        "clocks": main["clocks"],
        "calls": main["calls"],
        "hard": hard,
    })
    if train:
        out.update({"timing": train["timing"], "eager_ms_per_step": train["eager_ms_per_step"],
                    "calls_event_floor_ms": train["calls_event_floor_ms"],
                    "roofline_by_call": train["roofline_by_call"], "step_hbm": train["step_hbm"],
                    "wall_s_timed_loop": train["wall_s_timed_loop"]})
    if wl.name in PAPER_CONTEXT:
        out["context"] = PAPER_CONTEXT[wl.name]
    if optimizer:
        out["optimizer"] = optimizer
    if dp:
        out["dp_exchange"] = dp
    if e2e_train:
        out["e2e"] = e2e_train
    if e2e_hard:
        hard["e2e"] = e2e_hard
        if train is None:
            out["e2e"] = e2e_hard
    if not args.profile:
        out["fit"] = time_quantile_fit(wl, flush)
        out["pipe_rates"] = rates
    return out


def time_dp_exchange(st, world):
    """The data-parallel exchange of a training step (all-reduce of the
    gradients before the update), timed on its own: the fwd+bwd step has no
    collective."""
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
    return {"ms": ms_x, "collective": "NCCL all-reduce (sum) of the gradients, then / N",
            "bytes_per_rank": int(sum(g.numel() * 4 for g in grads))}


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


def measure_pipe_rates(sms: int, iters: int = 2048, reps: int = 5) -> dict:
    """Sustained issue rates of the instructions the kernels run, per SM and
    clock, from the library's throughput probe (one block of 1024 threads
    per SM, independent chains of one instruction kind, SM cycles read with
    clock64): the LOP3 mux with three varying registers ("mux3", the hard
    tree's upper levels), IMAD (its level 0), the two interleaved ("mix",
    the tree's instruction mix), the LOP3 mux with an invariant operand
    ("lop3") and FFMA (the soft kernels).  Median over blocks, then over
    `reps` launches."""
    import paper_2602_07400_gb300 as bl
    n = bl.bitlogic_issue_probe_threads()
    nb = bl.bitlogic_issue_probe_blocks()
    sink = torch.empty(n, dtype=torch.int32, device="cuda")
    cyc = torch.empty(nb, dtype=torch.int64, device="cuda")
    ops_per_block = (n // nb) * iters * bl.bitlogic_issue_probe_ops_per_iter()
    _, sm_max, _ = peaks()
    out = {"sms": sms, "probe": "independent dependency chains, one block of 1024 threads per SM, "
                                "SM cycles from clock64; median over blocks and 5 launches"}
    for kind in ("mux3", "imad", "mix", "lop3", "ffma"):
        bl.bitlogic_issue_probe(kind, iters, sink, cyc)
        per = []
        for _ in range(reps):
            bl.bitlogic_issue_probe(kind, iters, sink, cyc)
            c = cyc.cpu().numpy().astype(np.float64)
            per.append(float(np.median(ops_per_block / c)))
        r = float(np.median(per))
        out[kind] = {"lane_ops_per_sm_per_clk": round(r, 2),
                     "T_lane_ops_s_at_max_clock": round(r * sms * sm_max * 1e6 / 1e12, 3)}
    return out


def hard_roofline(roof: dict, rates: dict, sms: int, clocks: dict) -> dict:
    """The hard layer against the rate at which this GPU issues its
    instruction mix.  The mux tree is integer work only (IMAD at level 0,
    three-register LOP3 muxes above), and no integer instruction stream
    issues at the FP32 lanes' rate: the measured rate of IMAD and the mux
    interleaved one to one, per SM and clock, times the SMs and the median
    SM clock sampled while the kernel ran, is the peak.  The fraction against
    the issue rate of 128 lanes per SM and clock stays beside it."""
    mhz = clocks.get("sm_mhz") or clocks.get("sm_max_mhz") or 2070.0
    mix = rates["mix"]["lane_ops_per_sm_per_clk"]
    out = dict(roof)
    out["frac_issue_rate"] = roof["frac"]
    out["peak_issue_rate"] = roof["peak"]
    out["peak"] = mix * sms * mhz * 1e6 / 1e12
    out["frac"] = roof["achieved"] / out["peak"]
    out["achieved_per_sm_per_clk"] = roof["achieved"] * 1e12 / (sms * mhz * 1e6)
    out["unit"] = "Tops/s (mux operations against the measured IMAD + LOP3 mux issue rate)"
    out["peak_source"] = (f"issue probe in this run: IMAD and three-register LOP3 interleaved 1:1, "
                          f"{mix:.1f} lane-ops per SM and clock x {sms} SMs x {mhz:.0f} MHz (median SM clock "
                          f"sampled during the timed loop); issue-rate peak (128 lanes per SM and clock) in "
                          f"peak_issue_rate")
    out.pop("frac_at_sampled_clock", None)
    return out


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


def cpu_baseline_train(wl, budget_s=12.0, node="soft"):
    import oracle
    cores = oracle.max_threads()
    r, n = calibrated(lambda w_, n_, seed=0: oracle_train_rate(w_, n_, seed, node), wl, budget_s, 4, wl.batch)
    return {"value": r, "unit": "samples/s", "cores": cores, "kind": "oracle",
            "sample": f"train step (fwd+bwd) on {n} of the {wl.batch} samples of a batch, "
                      f"full {wl.widths[0]} x {wl.widths[1]} network, fp64, OpenMP over independent outputs"}


def cpu_baseline_hard(wl, budget_s=6.0):
    import oracle
    cores = oracle.max_threads()
    rh, nh = calibrated(oracle_hard_rate, wl, budget_s, 32, 1 << 16)
    return {"value": rh / 1e6, "unit": "MSamples/s", "cores": cores, "kind": "oracle",
            "sample": f"hard pass (encode+pack, 2 layers, popcount head) on {nh} of the {wl.batch} samples"}


def _reference_rate(fn, wl, lo, steps, warmup, per_step_s, calib_n):
    """Oracle rate over `steps` bounded samples of the workload (each about
    per_step_s of work) after `warmup` small ones."""
    r0 = fn(wl, min(wl.batch, calib_n))
    n = max(lo, int(r0 * per_step_s) // lo * lo)
    n = min(n, wl.batch)
    for i in range(warmup):
        fn(wl, lo, seed=100 + i)
    tot_s, tot_n = 0.0, 0
    for i in range(steps):
        r = fn(wl, n, seed=i)
        tot_s += n / r
        tot_n += n
    return tot_n / tot_s, n, tot_s


def run_reference(args):
    """The oracle as it stands on the host cores, on the same workloads,
    metric and unit as the GPU arm (each step a bounded sample)."""
    world, rank, _ = dist_env()
    if rank != 0:
        return None
    import oracle
    cores = oracle.max_threads()
    K, W = args.steps, args.warmup
    train_fn = lambda w_, n_, seed=0: oracle_train_rate(w_, n_, seed, args.node)  # noqa: E731
    out = {"impl": "reference"}
    out.update(base_line(world, K, W))
    out["dtype"] = "f64"
    if args.workload is None:
        # about 90 s of training-step oracle work and 30 s of hard-pass work
        wl = synth.WORKLOADS[HEADLINE_TRAIN]
        wh = synth.WORKLOADS[HEADLINE_HARD]
        v, n, tot = _reference_rate(train_fn, wl, 2, K, W, min(3.0, 90.0 / max(1, K + W)), 8)
        vh, nh, _ = _reference_rate(oracle_hard_rate, wh, 32, K, W, min(1.0, 30.0 / max(1, K + W)), 4096)
        out.update({"value": v, "unit": "samples/s", "ms_per_step": 1e3 * tot / max(1, K),
                    "config": {"workload": wl.name, "batch_per_gpu": wl.batch},
                    "cpu_baseline": {"value": v, "unit": "samples/s", "cores": cores, "kind": "oracle",
                                     "sample": f"{n} samples of the workload per step (the plain C oracle, "
                                               f"train fwd+bwd)"},
                    "e2e": {"value": v, "unit": "samples/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
                    "hard": {"value": vh / 1e6, "unit": "MSamples/s", "config": {"workload": wh.name,
                                                                                "batch_per_gpu": wh.batch},
                             "cpu_baseline": {"value": vh / 1e6, "unit": "MSamples/s", "cores": cores,
                                              "kind": "oracle",
                                              "sample": f"{nh} samples of the workload per step (hard pass)"}}})
        return out
    wl = synth.WORKLOADS[args.workload]
    hard_only = wl.name.startswith("hard_")
    fn = oracle_hard_rate if hard_only else train_fn
    lo = 32 if hard_only else 2
    # size one step so that the whole run (warm-up and timed steps) takes
    # about two minutes of oracle work, at most 1.5 s per step
    v, n, tot = _reference_rate(fn, wl, lo, K, W, min(1.5, 120.0 / max(1, K + W)), 4096 if hard_only else 64)
    unit = "samples/s"
    if hard_only:
        v /= 1e6
        unit = "MSamples/s"
    out.update({"value": v, "unit": unit, "ms_per_step": 1e3 * tot / max(1, K),
                "config": {"workload": wl.name, "batch_per_gpu": wl.batch},
                "cpu_baseline": {"value": v, "unit": unit, "cores": cores, "kind": "oracle",
                                 "sample": f"{n} samples of the workload per step (the plain C oracle, "
                                           f"{'hard pass' if hard_only else 'train fwd+bwd'})"},
                "e2e": {"value": v, "unit": unit, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}})
    return out


def main():
    args = parse_args()
    if args.impl == "reference":
        res = run_reference(args)
        if res is not None:
            print(json.dumps(res), flush=True)
        return
    world, rank, local = dist_env()
    torch.cuda.set_device(local)
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
    import paper_2602_07400_gb300 as bl
    bl.load()
    res = run_headline(args) if args.workload is None else run_single(args)
    if world > 1:
        torch.distributed.barrier()
        torch.distributed.destroy_process_group()
    if res is None:
        return
    if not args.profile and not args.no_cpu_baseline:
        if args.workload is None:
            res["cpu_baseline"] = cpu_baseline_train(synth.WORKLOADS[HEADLINE_TRAIN], node=args.node)
            res["hard"]["cpu_baseline"] = cpu_baseline_hard(synth.WORKLOADS[HEADLINE_HARD])
        else:
            wl = synth.WORKLOADS[args.workload]
            if not wl.name.startswith("hard_"):
                res["cpu_baseline"] = cpu_baseline_train(wl, node=args.node)
            res["hard"]["cpu_baseline"] = cpu_baseline_hard(wl)
            if wl.name.startswith("hard_"):
                res["cpu_baseline"] = res["hard"]["cpu_baseline"]
    print(json.dumps(res), flush=True)


if __name__ == "__main__":
    main()
