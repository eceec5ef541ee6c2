"""The hot path as call sequences over device-resident buffers.

``TrainStep`` runs one soft training step of the two-layer network of the
paper's protocol (§4 "Architecture": encoder -> logic layer -> logic layer
-> head): thermometer encode, two LUT forwards, group-sum head with
cross-entropy, two LUT backwards.  ``HardInfer`` runs the hard bit-packed
evaluation (App. C.1): binarize tables, encode + pack, hard layer 1, hard
layer 2 with the fused popcount head and argmax.  Buffers are allocated once
(torch provides the device memory); every step only enqueues library calls
on the current stream, so a step can be captured once as a CUDA graph and
replayed (``capture``), which removes the host work between the launches.
"""
from __future__ import annotations

from typing import Optional, Sequence

import numpy as np
import torch

from . import (NODE_FORMS, bitlogic_adamw_update, bitlogic_binarize_tables, bitlogic_build_csr,
               bitlogic_csr_positions, bitlogic_csr_reduce, bitlogic_pixel_histogram, bitlogic_quantile_thresholds,
               bitlogic_encode_thermometer, bitlogic_hard_forward, bitlogic_head_loss_ex,
               bitlogic_head_loss_workspace, bitlogic_lut_backward_node, bitlogic_lut_backward_through,
               bitlogic_lut_backward_u8, bitlogic_lut_forward_node,
               bitlogic_pack_bits, bitlogic_route_backward, bitlogic_route_backward_u8, bitlogic_route_forward,
               bitlogic_route_forward_u8, bitlogic_route_snap, bitlogic_encode_thermometer_u8,
               bitlogic_lut_forward_u8, bitlogic_encode_thermometer_bitrows, bitlogic_lut_forward_bitrows,
               bitlogic_lut_backward_bitrows, bitrow_words, bitlogic_degree_order)


def _nomark(name: str) -> None:
    return None


def fit_quantile_thresholds(batches, b: int, stream=None) -> list:
    """Quantile thermometer thresholds fitted on the pixels of every batch
    (uint8 CUDA tensors, e.g. the training split in pieces): one device
    histogram over all of them, read back once."""
    hist = None
    for x in batches:
        if hist is None:
            hist = torch.zeros(256, dtype=torch.int64, device=x.device)
        bitlogic_pixel_histogram(x, hist, stream)
    if hist is None:
        raise ValueError("no batches to fit")
    return [int(t) for t in bitlogic_quantile_thresholds(hist, b)]


def capture_graph(fn) -> torch.cuda.CUDAGraph:
    """Record ``fn()`` (library calls on the current stream) as a CUDA graph:
    one warm-up call on a side stream first (lazy set-up such as kernel
    attributes happens outside the capture), then the captured call.  Replay
    with ``graph.replay()``; the graph stays bound to the buffers ``fn`` used."""
    side = torch.cuda.Stream()
    side.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(side):
        fn()
    torch.cuda.current_stream().wait_stream(side)
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph):
        fn()
    return graph


def allreduce_gradients(grads, group=None) -> None:
    """Data-parallel exchange of a training step (the batch is sharded over
    ranks, every rank holds the whole network): sum
    the ranks' gradients and divide by the number of ranks, in place, one
    all-reduce per tensor in list order.  Each rank's loss is the mean over
    its own batch, so with equal batches the result is the gradient of the
    mean loss over all ranks' samples; every rank then applies the same
    update."""
    import torch.distributed as dist
    world = dist.get_world_size(group)
    for g in grads:
        dist.all_reduce(g, op=dist.ReduceOp.SUM, group=group)
        if world > 1:
            g.div_(world)


class Prefetcher:
    """Runs a step object (TrainStep, RoutedTrainStep or HardInfer) over
    host batches with the host-to-device copy of the next batch overlapping
    the current step: two device input buffers, each with its own captured
    graph of the step, and a copy stream.  ``prefetch`` enqueues a batch's
    copy; ``run`` replays the step on the oldest fetched batch and copies its
    result (the attribute ``out``) into a host tensor, all asynchronously."""

    def __init__(self, step, names=("x", "labels"), out="loss", capture=None):
        self.step, self.names, self.out = step, tuple(names), out
        # the buffers start as copies of the step's current inputs, so the
        # warm-up run of each capture reads valid data (labels in range)
        self.bufs = [{n: getattr(step, n).clone() for n in self.names} for _ in range(2)]
        self.graphs = []
        for b in range(2):
            for n in self.names:
                setattr(step, n, self.bufs[b][n])
            self.graphs.append(capture() if capture is not None else step.capture())
        self.copy_stream = torch.cuda.Stream()
        self.copied = [torch.cuda.Event() for _ in range(2)]
        self.consumed = [torch.cuda.Event() for _ in range(2)]
        self.n_fetched = 0
        self.n_run = 0

    def start(self):
        """Order the copy stream after the work already on the current stream."""
        self.copy_stream.wait_stream(torch.cuda.current_stream())

    def prefetch(self, host: dict):
        b = self.n_fetched % 2
        cs = self.copy_stream
        cs.wait_event(self.consumed[b])   # the step that last read buffer b is done
        with torch.cuda.stream(cs):
            for n in self.names:
                self.bufs[b][n].copy_(host[n], non_blocking=True)
        self.copied[b].record(cs)
        self.n_fetched += 1

    def run(self, out_host: torch.Tensor):
        b = self.n_run % 2
        cur = torch.cuda.current_stream()
        cur.wait_event(self.copied[b])
        self.graphs[b].replay()
        out_host.copy_(getattr(self.step, self.out), non_blocking=True)
        self.consumed[b].record(cur)
        self.n_run += 1


class Network:
    """Connectivity, table logits and inverse connectivity of a two-layer
    LUT network, resident on the device."""

    def __init__(self, conn1: np.ndarray, theta1: np.ndarray, conn2: np.ndarray,
                 theta2: np.ndarray, w_in: int, device="cuda"):
        self.w_in = int(w_in)
        self.w1, self.k1 = conn1.shape
        self.w2, self.k2 = conn2.shape
        dev = torch.device(device)
        self.conn1 = torch.from_numpy(np.ascontiguousarray(conn1, np.int32)).to(dev)
        self.conn2 = torch.from_numpy(np.ascontiguousarray(conn2, np.int32)).to(dev)
        self.theta1 = torch.from_numpy(np.ascontiguousarray(theta1, np.float32)).to(dev)
        self.theta2 = torch.from_numpy(np.ascontiguousarray(theta2, np.float32)).to(dev)
        off1, edge1 = bitlogic_build_csr(conn1, self.w_in)
        off2, edge2 = bitlogic_build_csr(conn2, self.w1)
        self.off1, self.edge1 = torch.from_numpy(off1).to(dev), torch.from_numpy(edge1).to(dev)
        self.off2, self.edge2 = torch.from_numpy(off2).to(dev), torch.from_numpy(edge2).to(dev)
        # CSR position of every edge: the per-edge gradient terms are stored
        # in CSR order, so each input's terms are one contiguous block
        self.pos1 = torch.from_numpy(bitlogic_csr_positions(edge1)).to(dev)
        self.pos2 = torch.from_numpy(bitlogic_csr_positions(edge2)).to(dev)
        # layer-1 nodes by decreasing consumer count: the order in which the
        # layer-1 backward on wire bit rows takes them (the longest first),
        # with layer 2's CSR map in that order's sequence (node order1[p]'s
        # edges at positions off2o[p] .. off2o[p+1] - 1; layer 2 stores its
        # terms at those positions for that backward)
        order1 = bitlogic_degree_order(off2)
        rank = np.empty_like(order1)
        rank[order1] = np.arange(self.w1, dtype=np.int32)
        off2o, edge2o = bitlogic_build_csr(rank[np.ascontiguousarray(conn2, np.int32)], self.w1)
        self.order1 = torch.from_numpy(order1).to(dev)
        self.off2o, self.edge2o = torch.from_numpy(off2o).to(dev), torch.from_numpy(edge2o).to(dev)
        self.pos2o = torch.from_numpy(bitlogic_csr_positions(edge2o)).to(dev)


# On fp32 wires, per-edge input-gradient terms larger than this are summed by
# the layer-1 backward itself instead of a separate CSR reduction (measured
# faster on GB300 for the CIFAR-shaped layers, 1.6 and 6.3 GB of terms, and
# slower for the MNIST-shaped one, 0.2 GB).  On byte wires the layer-1
# backward always sums them (MNIST shape: 0.216 against 0.2235 ms per step).
FUSE_DY1_TERM_BYTES = 512 << 20


class TrainStep:
    """One soft training step.  The backward is fused across the call
    boundaries the ABI offers: the head emits one gradient row per class
    (``dyg``) that the layer-2 backward reads for every node of the class.
    Layer 1's output gradient (the input gradient of layer 2) takes one of
    three routes:

    * ``through`` (default when layer 2's fan-in is at most 3): the layer-1
      backward recomputes it from layer 2's connectivity, tables and output
      gradient rows (bitlogic_lut_backward_through), so layer 2 needs only
      its table gradient and nothing per edge is stored;
    * ``fuse_dy1`` (default on byte wires, and on fp32 wires when layer 2's
      per-edge terms exceed FUSE_DY1_TERM_BYTES): layer 2 stores its per-edge
      terms and the layer-1 backward sums them through the CSR map on the fly;
    * otherwise a CSR reduction of the terms into ``dy1``, which the
      dtheta-only layer-1 backward reads.

    Layer 1 reads the encoder's wires as bytes (``bytes1``, the default when
    B % 4 == 0 and no layer-1 input gradient is wanted): its inputs are
    binary, so every corner weight of the relaxed table is 0 or 1 and the
    layer-1 forward is a table lookup (bitlogic_lut_forward_u8) and its table
    gradient adds each sample's gradient to the one entry the sample selects
    (bitlogic_lut_backward_u8 / _through on byte rows); the encoder then
    writes byte rows only, and ``bits`` is that uint8 tensor.  The table
    gradient equals the fp32-row form bit for bit; the forward returns the
    table entry itself, which the fp32 lerp tree reaches up to rounding.
    With ``bits1`` (the default on byte wires off the through route) the
    wires are kept at one bit per sample instead, an eighth of the bytes (the
    CIFAR-100-shaped layer input then stays in L2):
    bitlogic_encode_thermometer_bitrows writes them and the layer-1 kernels
    read those words (bitlogic_lut_forward_bitrows / _backward_bitrows) with
    the same results bit for bit; ``bits`` is then the int32 tensor of words
    and ``wires()`` writes the wires out as bytes on demand.  Set
    ``keep_dy1`` to also write dY1 (e.g. to check it).  ``node`` picks the
    LightLUT form of both layers: "soft", or "st" (hard table samples in the
    forward, straight-through gradient to the logits)."""

    def __init__(self, net: Network, B: int, d: int, thresholds: Sequence[int], C: int,
                 tau: float, want_dx1: bool = False, keep_dy1: bool = False,
                 fuse_dy1: Optional[bool] = None, csr_order: bool = True, node: str = "soft",
                 through: Optional[bool] = None, bytes1: Optional[bool] = None,
                 bits1: Optional[bool] = None, device="cuda"):
        dev = torch.device(device)
        if node not in NODE_FORMS:
            raise ValueError(f"node must be one of {sorted(NODE_FORMS)}")
        self.node = node
        self.net, self.B, self.d, self.C, self.tau = net, int(B), int(d), int(C), float(tau)
        self.thr = [int(t) for t in thresholds]
        assert d * len(self.thr) == net.w_in
        assert net.w2 % C == 0
        if through is None:
            through = net.k2 <= 3 and B % 4 == 0 and not want_dx1
        if through and (net.k2 > 3 or B % 4 != 0 or want_dx1):
            raise ValueError("the through route needs layer-2 fan-in <= 3, B % 4 == 0 and no layer-1 input gradient")
        self.through = bool(through)
        if bytes1 is None:
            bytes1 = B % 4 == 0 and not want_dx1
        if fuse_dy1 is None:
            # on byte wires the layer-1 backward streams the terms itself
            # (faster than the CSR reduction at every measured shape); on fp32
            # wires the separate reduction wins below FUSE_DY1_TERM_BYTES
            fuse_dy1 = bool(bytes1) or 4 * net.w2 * net.k2 * B > FUSE_DY1_TERM_BYTES
        f32 = dict(dtype=torch.float32, device=dev)
        self.x = torch.zeros(B, d, dtype=torch.uint8, device=dev)
        self.labels = torch.zeros(B, dtype=torch.int32, device=dev)
        self.y1 = torch.empty(net.w1, B, **f32)
        self.y2 = torch.empty(net.w2, B, **f32)
        self.logits = torch.empty(B, C, **f32)
        self.loss = torch.zeros(1, **f32)
        self.dyg = torch.empty(C, B, **f32)          # gradient row shared by each class's nodes
        self.fuse_dy1 = bool(fuse_dy1) and not self.through
        if bytes1 and (B % 4 != 0 or want_dx1):
            raise ValueError("byte wires for layer 1 need B % 4 == 0 and no layer-1 input gradient")
        self.bytes1 = bool(bytes1)
        if bits1 is None:
            bits1 = self.bytes1 and not self.through
        if bits1 and not (self.bytes1 and not self.through):
            raise ValueError("wire bit rows need byte wires for layer 1 and a route other than through")
        self.bits1 = bool(bits1)
        # the encoder's output: wire bit rows (bits1), byte rows (bytes1) or
        # fp32 rows
        if self.bits1:
            self.bits = torch.empty(net.w_in, bitrow_words(B), dtype=torch.int32, device=dev)
        else:
            self.bits = torch.empty(net.w_in, B, dtype=torch.uint8 if self.bytes1 else torch.float32, device=dev)
        # per-edge terms stored in CSR order (each input's terms contiguous,
        # read without the edge map) instead of edge order
        self.csr_order = bool(csr_order)
        self.dy1 = torch.empty(net.w1, B, **f32) if (keep_dy1 or not (self.fuse_dy1 or self.through)) else None
        self.dth1 = torch.empty_like(net.theta1)
        self.dth2 = torch.empty_like(net.theta2)
        self.dbits = torch.empty(net.w_in, B, **f32) if want_dx1 else None
        # per-edge input-gradient terms of layer 2 (and of layer 1 when its
        # input gradient is wanted)
        self.edges2 = None if self.through else torch.empty(net.w2 * net.k2, B, **f32)
        self.edges1 = torch.empty(net.w1 * net.k1, B, **f32) if want_dx1 else None
        self.ws_head = torch.empty(bitlogic_head_loss_workspace(B, C), dtype=torch.uint8, device=dev)

    def load(self, x: torch.Tensor, labels: torch.Tensor, non_blocking: bool = False):
        self.x.copy_(x, non_blocking=non_blocking)
        self.labels.copy_(labels, non_blocking=non_blocking)

    def forward(self, stream=None, mark=_nomark):
        n = self.net
        if self.bits1:
            bitlogic_encode_thermometer_bitrows(self.x, self.thr, self.bits, stream)
            mark("encode")
            bitlogic_lut_forward_bitrows(self.bits, self.B, n.conn1, n.theta1, self.y1, self.node, stream)
        elif self.bytes1:
            bitlogic_encode_thermometer_u8(self.x, self.thr, self.bits, stream)
            mark("encode")
            bitlogic_lut_forward_u8(self.bits, n.conn1, n.theta1, self.y1, self.node, stream)
        else:
            bitlogic_encode_thermometer(self.x, self.thr, self.bits, stream)
            mark("encode")
            bitlogic_lut_forward_node(self.bits, n.conn1, n.theta1, self.y1, self.node, stream)
        mark("forward1")
        bitlogic_lut_forward_node(self.y1, n.conn2, n.theta2, self.y2, self.node, stream)
        mark("forward2")
        bitlogic_head_loss_ex(self.y2, self.labels, self.C, self.tau, self.loss, self.ws_head,
                              logits=self.logits, dY_grouped=self.dyg, stream=stream)
        mark("head")

    def backward(self, stream=None, mark=_nomark):
        n = self.net
        co = self.csr_order
        nd = self.node
        g = n.w2 // self.C
        if self.through:
            # layer 2: table gradient only; layer 1: its output gradient
            # recomputed through layer 2 inside its table-gradient kernel
            bitlogic_lut_backward_node(self.y1, n.conn2, n.theta2, self.dth2, nd, dY=self.dyg, dy_group=g,
                                       stream=stream)
            mark("backward2")
            bitlogic_lut_backward_through(self.bits, n.conn1, n.theta1, self.dth1,
                                          self.y1, n.conn2, n.theta2, self.dyg, g, n.off2, n.edge2, node=nd,
                                          dY_out=self.dy1, stream=stream)
            mark("backward1")
            return
        # the bit-row layer-1 backward reads the terms through the CSR map in
        # its node order; every other consumer through the map in node order
        ordered = self.fuse_dy1 and self.bits1
        bitlogic_lut_backward_node(self.y1, n.conn2, n.theta2, self.dth2, nd, dY=self.dyg,
                                   dy_group=g, edge_terms=self.edges2,
                                   edge_pos=(n.pos2o if ordered else n.pos2) if co else None, stream=stream)
        mark("backward2")
        pos1 = n.pos1 if (co and self.edges1 is not None) else None
        edge2 = None if co else n.edge2
        if ordered:
            bitlogic_lut_backward_bitrows(self.bits, self.B, n.conn1, n.theta1, self.dth1, nd, up_terms=self.edges2,
                                          up_off=n.off2o, up_edge=None if co else n.edge2o, dY_out=self.dy1,
                                          order=n.order1, stream=stream)
        elif self.fuse_dy1 and self.bytes1:
            bitlogic_lut_backward_u8(self.bits, n.conn1, n.theta1, self.dth1, nd, up_terms=self.edges2,
                                     up_off=n.off2, up_edge=edge2, dY_out=self.dy1, stream=stream)
        elif self.fuse_dy1:
            bitlogic_lut_backward_node(self.bits, n.conn1, n.theta1, self.dth1, nd, up_terms=self.edges2,
                                       up_off=n.off2, up_edge=edge2, edge_terms=self.edges1,
                                       edge_pos=pos1, dY_out=self.dy1, stream=stream)
        else:
            bitlogic_csr_reduce(self.edges2, n.off2, edge2, self.dy1, stream)
            mark("csr2")
            if self.bits1:
                bitlogic_lut_backward_bitrows(self.bits, self.B, n.conn1, n.theta1, self.dth1, nd, dY=self.dy1,
                                              stream=stream)
            elif self.bytes1:
                bitlogic_lut_backward_u8(self.bits, n.conn1, n.theta1, self.dth1, nd, dY=self.dy1, stream=stream)
            else:
                bitlogic_lut_backward_node(self.bits, n.conn1, n.theta1, self.dth1, nd, dY=self.dy1,
                                           edge_terms=self.edges1, edge_pos=pos1, stream=stream)
        mark("backward1")
        if self.dbits is not None:
            bitlogic_csr_reduce(self.edges1, n.off1, None if co else n.edge1, self.dbits, stream)
            mark("csr1")

    def run(self, stream=None, mark=_nomark):
        self.forward(stream, mark)
        self.backward(stream, mark)

    def wires(self, stream=None) -> torch.Tensor:
        """Layer 1's input wires [w_in, B]: ``bits``, or under ``bits1`` the
        thermometer of the loaded samples written out as bytes into a new
        tensor."""
        if not self.bits1:
            return self.bits
        out = torch.empty(self.net.w_in, self.B, dtype=torch.uint8, device=self.bits.device)
        bitlogic_encode_thermometer_u8(self.x, self.thr, out, stream)
        return out

    def capture(self) -> torch.cuda.CUDAGraph:
        """One run() (forward + backward) as a CUDA graph: a replay launches
        the same kernels with no host work between them."""
        return capture_graph(self.run)

    def gradients(self):
        """The tensors a data-parallel step exchanges before the update."""
        return [self.dth1, self.dth2]

    def update(self, lr: float = 0.01, betas=(0.9, 0.999), eps: float = 1e-8,
               weight_decay: float = 0.0, stream=None, mark=_nomark):
        """AdamW step on both layers' table logits from the last backward
        (§4 "Training": the paper's settings are the defaults); the moment
        buffers start at zero on the first call."""
        n = self.net
        if not hasattr(self, "opt_m1"):
            self.opt_m1, self.opt_v1 = torch.zeros_like(n.theta1), torch.zeros_like(n.theta1)
            self.opt_m2, self.opt_v2 = torch.zeros_like(n.theta2), torch.zeros_like(n.theta2)
            self.opt_step = 0
        self.opt_step += 1
        bitlogic_adamw_update(n.theta1, self.opt_m1, self.opt_v1, self.dth1, self.opt_step, lr, betas, eps,
                              weight_decay, stream)
        bitlogic_adamw_update(n.theta2, self.opt_m2, self.opt_v2, self.dth2, self.opt_step, lr, betas, eps,
                              weight_decay, stream)
        mark("update")

    # kernels one run() launches: encode 1, forwards 2, head 2, backwards 2
    # (+ the CSR reduction of layer 2's terms unless fused or recomputed, +
    # the layer-1 CSR reduction when the input gradient is wanted)
    @property
    def kernels_per_run(self) -> int:
        return 7 + (0 if (self.fuse_dy1 or self.through) else 1) + (1 if self.dbits is not None else 0)


class RoutedNetwork:
    """A two-layer LUT network with learnable routing (§3 "Connectivity"):
    per node slot a candidate pool (int32 [w*k, Kc]) and routing logits
    (fp32 [w*k, Kc], zero at initialisation), plus the table logits.  The
    nodes read their slot inputs through the identity connectivity."""

    def __init__(self, cand1: np.ndarray, r1: np.ndarray, theta1: np.ndarray, cand2: np.ndarray,
                 r2: np.ndarray, theta2: np.ndarray, w_in: int, device="cuda"):
        dev = torch.device(device)
        self.w_in = int(w_in)
        self.w1, K1 = theta1.shape
        self.w2, K2 = theta2.shape
        self.k1, self.k2 = K1.bit_length() - 1, K2.bit_length() - 1
        self.Kc = cand1.shape[1]
        assert cand1.shape == (self.w1 * self.k1, self.Kc) and cand2.shape == (self.w2 * self.k2, self.Kc)
        t = lambda a, dt: torch.from_numpy(np.ascontiguousarray(a, dt)).to(dev)
        self.cand1, self.cand2 = t(cand1, np.int32), t(cand2, np.int32)
        self.r1, self.r2 = t(r1, np.float32), t(r2, np.float32)
        self.theta1, self.theta2 = t(theta1, np.float32), t(theta2, np.float32)
        self.ident1 = torch.arange(self.w1 * self.k1, dtype=torch.int32, device=dev).view(self.w1, self.k1)
        self.ident2 = torch.arange(self.w2 * self.k2, dtype=torch.int32, device=dev).view(self.w2, self.k2)
        # candidate CSR of layer 2 (its input gradient feeds layer 1)
        off2, edge2 = bitlogic_build_csr(np.ascontiguousarray(cand2, np.int32), self.w1)
        self.coff2, self.cedge2 = t(off2, np.int32), t(edge2, np.int32)

    def snap(self) -> "Network":
        """The discretized network: each slot keeps its most likely candidate."""
        conns = []
        for cand, r, w, k in ((self.cand1, self.r1, self.w1, self.k1), (self.cand2, self.r2, self.w2, self.k2)):
            conn = torch.empty(w * k, dtype=torch.int32, device=cand.device)
            bitlogic_route_snap(cand, r, conn)
            conns.append(conn.view(w, k).cpu().numpy())
        return Network(conns[0], self.theta1.cpu().numpy(), conns[1], self.theta2.cpu().numpy(), self.w_in,
                       device=self.cand1.device)


class RoutedTrainStep:
    """One training step of a RoutedNetwork: encode, per layer the routing
    (slot inputs as the expected selection) and the LUT nodes over them,
    head, and the backward through nodes and routing (gradients of the
    table and routing logits).  The encoder's wires are kept as bytes: the
    layer-1 routing gathers them from a quarter of the memory."""

    def __init__(self, net: RoutedNetwork, B: int, d: int, thresholds: Sequence[int], C: int, tau: float,
                 node: str = "soft", device="cuda"):
        dev = torch.device(device)
        if node not in NODE_FORMS:
            raise ValueError(f"node must be one of {sorted(NODE_FORMS)}")
        self.net, self.B, self.d, self.C, self.tau, self.node = net, int(B), int(d), int(C), float(tau), node
        self.thr = [int(t) for t in thresholds]
        assert d * len(self.thr) == net.w_in and net.w2 % C == 0
        f32 = dict(dtype=torch.float32, device=dev)
        s1, s2 = net.w1 * net.k1, net.w2 * net.k2
        self.x = torch.zeros(B, d, dtype=torch.uint8, device=dev)
        self.labels = torch.zeros(B, dtype=torch.int32, device=dev)
        self.bits = torch.empty(net.w_in, B, dtype=torch.uint8, device=dev)   # 0/1 wires
        self.xr1, self.xr2 = torch.empty(s1, B, **f32), torch.empty(s2, B, **f32)
        self.p1, self.p2 = torch.empty(s1, net.Kc, **f32), torch.empty(s2, net.Kc, **f32)
        self.y1 = torch.empty(net.w1, B, **f32)
        self.y2 = torch.empty(net.w2, B, **f32)
        self.logits = torch.empty(B, C, **f32)
        self.loss = torch.zeros(1, **f32)
        self.dyg = torch.empty(C, B, **f32)
        self.g1, self.g2 = torch.empty(s1, B, **f32), torch.empty(s2, B, **f32)   # dL/dXr
        self.dy1 = torch.empty(net.w1, B, **f32)
        self.dth1, self.dth2 = torch.empty_like(net.theta1), torch.empty_like(net.theta2)
        self.dr1, self.dr2 = torch.empty_like(net.r1), torch.empty_like(net.r2)
        self.ws_head = torch.empty(bitlogic_head_loss_workspace(B, C), dtype=torch.uint8, device=dev)

    def load(self, x: torch.Tensor, labels: torch.Tensor, non_blocking: bool = False):
        self.x.copy_(x, non_blocking=non_blocking)
        self.labels.copy_(labels, non_blocking=non_blocking)

    def forward(self, stream=None, mark=_nomark):
        n = self.net
        bitlogic_encode_thermometer_u8(self.x, self.thr, self.bits, stream)
        mark("encode")
        bitlogic_route_forward_u8(self.bits, n.cand1, n.r1, self.xr1, self.p1, stream)
        mark("route1")
        bitlogic_lut_forward_node(self.xr1, n.ident1, n.theta1, self.y1, self.node, stream)
        mark("forward1")
        bitlogic_route_forward(self.y1, n.cand2, n.r2, self.xr2, self.p2, stream)
        mark("route2")
        bitlogic_lut_forward_node(self.xr2, n.ident2, n.theta2, self.y2, self.node, stream)
        mark("forward2")
        bitlogic_head_loss_ex(self.y2, self.labels, self.C, self.tau, self.loss, self.ws_head,
                              logits=self.logits, dY_grouped=self.dyg, stream=stream)
        mark("head")

    def backward(self, stream=None, mark=_nomark):
        n = self.net
        # layer 2: node gradients per slot (identity connectivity: the edge
        # terms are dL/dXr2), then the routing: dr2 and dY1
        bitlogic_lut_backward_node(self.xr2, n.ident2, n.theta2, self.dth2, self.node, dY=self.dyg,
                                   dy_group=n.w2 // self.C, edge_terms=self.g2, stream=stream)
        mark("backward2")
        bitlogic_route_backward(self.y1, n.cand2, n.r2, self.g2, self.dr2, self.p2, n.coff2, n.cedge2,
                                self.dy1, stream)
        mark("route_bwd2")
        bitlogic_lut_backward_node(self.xr1, n.ident1, n.theta1, self.dth1, self.node, dY=self.dy1,
                                   edge_terms=self.g1, stream=stream)
        mark("backward1")
        bitlogic_route_backward_u8(self.bits, n.cand1, n.r1, self.g1, self.dr1, stream)
        mark("route_bwd1")

    def run(self, stream=None, mark=_nomark):
        self.forward(stream, mark)
        self.backward(stream, mark)

    def capture(self) -> torch.cuda.CUDAGraph:
        return capture_graph(self.run)

    def gradients(self):
        return [self.dth1, self.dth2, self.dr1, self.dr2]

    def update(self, lr: float = 0.01, betas=(0.9, 0.999), eps: float = 1e-8, weight_decay: float = 0.0,
               stream=None, mark=_nomark):
        """AdamW (§4 settings) on the table and routing logits of both layers."""
        n = self.net
        params = ((n.theta1, self.dth1), (n.theta2, self.dth2), (n.r1, self.dr1), (n.r2, self.dr2))
        if not hasattr(self, "opt_state"):
            self.opt_state = [(torch.zeros_like(p), torch.zeros_like(p)) for p, _ in params]
            self.opt_step = 0
        self.opt_step += 1
        for (p, g), (m, v) in zip(params, self.opt_state):
            bitlogic_adamw_update(p, m, v, g, self.opt_step, lr, betas, eps, weight_decay, stream)
        mark("update")

    # encode 1, routing forwards 2, LUT forwards 2, head 2, LUT backwards 2,
    # routing dr 2, routing dX 1
    kernels_per_run = 12
    fuse_dy1 = False


class HardInfer:
    def __init__(self, net: Network, N: int, d: int, thresholds: Sequence[int], C: int,
                 keep_layer2: bool = False, device="cuda"):
        dev = torch.device(device)
        self.net, self.N, self.d, self.C = net, int(N), int(d), int(C)
        self.thr = [int(t) for t in thresholds]
        W = (N + 31) // 32
        i32 = dict(dtype=torch.int32, device=dev)
        self.x = torch.zeros(N, d, dtype=torch.uint8, device=dev)
        self.table1 = torch.empty(net.w1, dtype=torch.int64, device=dev)
        self.table2 = torch.empty(net.w2, dtype=torch.int64, device=dev)
        self.xp = torch.empty(net.w_in, W, **i32)
        self.yp1 = torch.empty(net.w1, W, **i32)
        self.yp2 = torch.empty(net.w2, W, **i32) if keep_layer2 else None
        self.counts = torch.empty(N, C, **i32)
        self.pred = torch.empty(N, **i32)

    def binarize(self, stream=None, mark=_nomark):
        bitlogic_binarize_tables(self.net.theta1, self.table1, stream)
        bitlogic_binarize_tables(self.net.theta2, self.table2, stream)
        mark("binarize")

    def run(self, stream=None, mark=_nomark):
        n = self.net
        bitlogic_pack_bits(self.x, self.thr, self.xp, stream)
        mark("pack")
        bitlogic_hard_forward(self.xp, self.N, n.conn1, self.table1, yp=self.yp1, stream=stream)
        mark("hard1")
        bitlogic_hard_forward(self.yp1, self.N, n.conn2, self.table2, yp=self.yp2, C=self.C,
                              counts=self.counts, pred=self.pred, stream=stream)
        mark("hard2")

    def capture(self, binarize: bool = True) -> torch.cuda.CUDAGraph:
        """One hard pass (with the table binarization when ``binarize``) as a
        CUDA graph."""
        def one():
            if binarize:
                self.binarize()
            self.run()
        return capture_graph(one)

    # kernels: binarize 2; pack 1, layer 1, layer 2 with head, argmax
    kernels_per_binarize = 2
    kernels_per_run = 4


def unpack_bits(words: torch.Tensor, N: int) -> np.ndarray:
    """int32 words [rows, W] (uint32 bit patterns) -> uint8 bits [rows, N] on the host."""
    w = words.detach().cpu().numpy().view(np.uint32)
    bits = (w[:, :, None] >> np.arange(32, dtype=np.uint32)[None, None, :]) & 1
    return bits.reshape(w.shape[0], -1)[:, :N].astype(np.uint8)
