"""Seeded synthetic inputs for the LUT-network hot path.

This module only draws random inputs of the right shapes and value
distributions; it holds none of the method's arithmetic (no encoding, no
node evaluation, no head).  Both the CUDA path and the CPU oracle consume
what it returns, so it is the one piece of code they share.

The real datasets of the paper (MNIST, Fashion-MNIST, CIFAR-10/100, §4
"Data") are not available; class-conditional Gaussian blobs of the same
shapes stand in for them:

* a class mean image ``mu_c`` with pixels uniform in [0, 255];
* a pixel ``clamp(round(mu_c[p] + sigma * z), 0, 255)`` with ``z ~ N(0, 1)``;
* a label uniform in ``0 .. C-1``.

Fixed connectivity draws ``k`` distinct input indices per node, uniformly
(the "random-unique" fixed routing of §3 and App. A "Initialization");
table logits are ``theta ~ N(0, 1)`` in fp32 (zero-mean Gaussian node
init, App. A "Initialization").
"""
from __future__ import annotations

import dataclasses
from typing import List, Optional, Tuple

import numpy as np
import torch


@dataclasses.dataclass(frozen=True)
class Workload:
    """Shapes of one synthetic workload (names follow the paper: d input
    features, b thresholds per feature, w nodes per layer, k fan-in,
    C classes, tau the group-sum temperature)."""

    name: str
    batch: int                 # B for training, N for hard inference
    d: int                     # raw uint8 features per sample
    classes: int               # C
    sigma: float               # blob pixel standard deviation
    thresholds: Tuple[int, ...]  # thermometer thresholds (uint8, ascending)
    widths: Tuple[int, int]    # nodes of layer 1 and layer 2
    k: int                     # fan-in of every node
    tau: float                 # group-sum temperature
    Kc: int = 0                # learnable routing: candidates per slot (0: fixed connectivity)

    @property
    def b(self) -> int:
        return len(self.thresholds)

    @property
    def w_in(self) -> int:
        return self.d * self.b

    @property
    def K(self) -> int:
        return 1 << self.k


def _even(n: int, b: int) -> Tuple[int, ...]:
    # literal equispaced thresholds 256*i/(b+1), i = 1..b, spelled out per
    # workload so that both sides receive them as input data
    return tuple(n * i for i in range(1, b + 1))


WORKLOADS = {
    # 256 samples, 784 features, thresholds {64,128,192}, 1000 x 1000, k=6
    "tiny": Workload("tiny", 256, 784, 10, 40.0, (64, 128, 192), (1000, 1000), 6, 10.0),
    # MNIST-shaped training throughput, 8000 x 8000, k=6 (and k=2)
    "mnist": Workload("mnist", 1024, 784, 10, 40.0, (64, 128, 192), (8000, 8000), 6, 20.0),
    "mnist_k2": Workload("mnist_k2", 1024, 784, 10, 40.0, (64, 128, 192), (8000, 8000), 2, 20.0),
    # fan-in 4, the rank the paper pins for its method comparisons (App. C.2)
    "mnist_k4": Workload("mnist_k4", 1024, 784, 10, 40.0, (64, 128, 192), (8000, 8000), 4, 20.0),
    # learnable routing with 16 candidates per slot in both layers, the
    # connectivity of the paper's best-of-space configuration (App. C.2), k=4
    "mnist_k4_routed16": Workload("mnist_k4_routed16", 1024, 784, 10, 40.0, (64, 128, 192), (8000, 8000), 4,
                                  20.0, Kc=16),
    # CIFAR-10-shaped: 3072 features, 7 thresholds -> 21504 bits, 64000 x 64000
    "cifar10": Workload("cifar10", 1024, 3072, 10, 50.0, _even(32, 7), (64000, 64000), 6, 50.0),
    # CIFAR-100-shaped wide: 15 thresholds -> 46080 bits, 128000 x 128000
    "cifar100": Workload("cifar100", 2048, 3072, 100, 50.0, _even(16, 15), (128000, 128000), 6, 100.0),
    # hard bit-packed inference on the CIFAR-10-shaped network, 2^22 samples
    "hard_cifar10": Workload("hard_cifar10", 1 << 22, 3072, 10, 50.0, _even(32, 7), (64000, 64000), 6, 50.0),
    # the shape of the paper's deployed MNIST network (§5 hardware
    # evaluation: w = 4000 per layer, n = 4, b = 4 thresholds -> 3136 bits,
    # popcount head 10 x 400) at its GPU batch of 1024 and at 2^22 samples;
    # equispaced thresholds stand in for the fitted quantile ones (the
    # throughput does not depend on the threshold values)
    "hard_mnist_w4000": Workload("hard_mnist_w4000", 1024, 784, 10, 40.0, _even(51, 4), (4000, 4000), 4, 40.0),
    "hard_mnist_w4000_4m": Workload("hard_mnist_w4000_4m", 1 << 22, 784, 10, 40.0, _even(51, 4), (4000, 4000),
                                    4, 40.0),
}


def class_means(C: int, d: int, seed: int) -> torch.Tensor:
    g = torch.Generator(device="cpu").manual_seed(seed)
    return torch.rand(C, d, generator=g, dtype=torch.float32) * 255.0


def blob_batch(n: int, d: int, C: int, sigma: float, seed: int,
               device: str | torch.device = "cpu",
               chunk: int = 1 << 16, means_seed: int | None = None) -> Tuple[torch.Tensor, torch.Tensor]:
    """Return ``(x, labels)``: ``x`` uint8 [n, d] (sample-major, as a raw
    image batch is stored) and ``labels`` int32 [n].  The class means come
    from ``means_seed`` (default: ``seed``); keep it fixed across batches to
    draw several batches of one synthetic dataset.  Data drawn on a CUDA
    device differ from data drawn on the CPU for the same seed; every
    comparison uses one draw, copied where needed."""
    device = torch.device(device)
    mu = class_means(C, d, seed if means_seed is None else means_seed).to(device)
    g = torch.Generator(device="cpu").manual_seed(seed + 1)
    labels = torch.randint(0, C, (n,), generator=g, dtype=torch.int64)
    labels_dev = labels.to(device)
    gz = torch.Generator(device=device).manual_seed(seed + 2)
    x = torch.empty(n, d, dtype=torch.uint8, device=device)
    for s0 in range(0, n, chunk):
        m = min(chunk, n - s0)
        z = torch.randn(m, d, generator=gz, device=device, dtype=torch.float32)
        v = mu.index_select(0, labels_dev[s0:s0 + m]).add_(z.mul_(sigma))
        x[s0:s0 + m] = v.round_().clamp_(0.0, 255.0).to(torch.uint8)
        del z, v
    return x, labels_dev.to(torch.int32)


def connectivity(w: int, k: int, w_in: int, seed: int) -> np.ndarray:
    """int32 [w, k]: k distinct indices in [0, w_in) per node, uniform."""
    if k > w_in:
        raise ValueError("fan-in larger than the layer input")
    rng = np.random.default_rng(seed)
    conn = rng.integers(0, w_in, size=(w, k), dtype=np.int64)
    while True:
        srt = np.sort(conn, axis=1)
        dup = np.any(srt[:, 1:] == srt[:, :-1], axis=1) if k > 1 else np.zeros(w, bool)
        rows = np.nonzero(dup)[0]
        if rows.size == 0:
            break
        conn[rows] = rng.integers(0, w_in, size=(rows.size, k), dtype=np.int64)
    return conn.astype(np.int32)


def candidate_pools(slots: int, Kc: int, w_in: int, seed: int) -> np.ndarray:
    """int32 [slots, Kc]: a uniformly drawn pool of Kc distinct inputs per
    node slot (learnable routing's candidate-pool mask, App. A)."""
    return connectivity(slots, Kc, w_in, seed)


def table_logits(w: int, K: int, seed: int, scale: float = 1.0) -> np.ndarray:
    """float32 [w, K] ~ N(0, scale^2)."""
    rng = np.random.default_rng(seed)
    return (rng.standard_normal((w, K), dtype=np.float32) * np.float32(scale)).astype(np.float32)


def uniform_activations(rows: int, B: int, seed: int) -> np.ndarray:
    """float32 [rows, B] uniform in [0, 1) (generic soft layer input)."""
    rng = np.random.default_rng(seed)
    return rng.random((rows, B), dtype=np.float32)


def binary_activations(rows: int, B: int, seed: int) -> np.ndarray:
    rng = np.random.default_rng(seed)
    return rng.integers(0, 2, size=(rows, B)).astype(np.float32)


def uniform_gradients(rows: int, B: int, seed: int, scale: float = 1.0) -> np.ndarray:
    rng = np.random.default_rng(seed)
    return (rng.standard_normal((rows, B), dtype=np.float32) * np.float32(scale)).astype(np.float32)


def random_words(rows: int, words: int, seed: int) -> np.ndarray:
    """uint32 [rows, words] of uniformly random bits."""
    rng = np.random.default_rng(seed)
    return rng.integers(0, 1 << 32, size=(rows, words), dtype=np.uint64).astype(np.uint32)


def random_tables(w: int, seed: int) -> np.ndarray:
    rng = np.random.default_rng(seed)
    return rng.integers(0, 1 << 63, size=(w,), dtype=np.uint64) * np.uint64(2) + \
        rng.integers(0, 2, size=(w,), dtype=np.uint64)


def routed_network(wl: Workload, seed: int = 0):
    """Candidate pools (layer 1 seed ``seed``, layer 2 ``seed + 1``), zero
    routing logits (App. A) and table logits of the routed network of ``wl``."""
    w1, w2 = wl.widths
    cand1 = candidate_pools(w1 * wl.k, wl.Kc, wl.w_in, seed)
    cand2 = candidate_pools(w2 * wl.k, wl.Kc, w1, seed + 1)
    r1 = np.zeros((w1 * wl.k, wl.Kc), np.float32)
    r2 = np.zeros((w2 * wl.k, wl.Kc), np.float32)
    th1 = table_logits(w1, wl.K, seed + 100)
    th2 = table_logits(w2, wl.K, seed + 101)
    return cand1, r1, th1, cand2, r2, th2


def network(wl: Workload, seed: int = 0):
    """Connectivity and table logits of the two-layer network of ``wl``
    (layer 1 connectivity seed ``seed``, layer 2 ``seed + 1``)."""
    w1, w2 = wl.widths
    conn1 = connectivity(w1, wl.k, wl.w_in, seed)
    conn2 = connectivity(w2, wl.k, w1, seed + 1)
    th1 = table_logits(w1, wl.K, seed + 100)
    th2 = table_logits(w2, wl.K, seed + 101)
    return conn1, th1, conn2, th2


def sample_positions(n: int, count: int, seed: int, must: Optional[List[int]] = None) -> np.ndarray:
    """Sorted distinct sample indices in [0, n) for sampled parity checks,
    always including the first and last sample (ragged tail)."""
    rng = np.random.default_rng(seed)
    pick = set([0, n - 1] + list(must or []))
    count = min(count, n)
    while len(pick) < count:
        pick.update(rng.integers(0, n, size=count - len(pick)).tolist())
    return np.array(sorted(pick), dtype=np.int64)
