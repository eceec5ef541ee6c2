"""GPU-vs-oracle parity of whole steps at the workloads' sizes, in the launch
configuration the benchmark times (``pipeline.TrainStep`` / ``HardInfer``).

* tiny (256 x 784, 1000 x 1000, k=6): every output element, including the
  input gradients of both layers.
* mnist (1024 x 784, 8000 x 8000, k=6 and k=2): every output element.
* cifar10 / cifar100 (64000- and 128000-wide layers, B = 1024 / 2048): every
  output element, the table gradients of both layers and layer 1's output
  gradient included.
* mnist_k4_routed16 (routed, 8000 x 8000, k = 4, 16 candidates): every
  output element, routing-logit gradients included.
* hard_cifar10 (2^22 samples): every sample recomputed by the oracle in
  chunks, bit-exact for the packed input, every layer-1 output word, the
  counts and the argmax.  hard_mnist_w4000_4m (2^22 samples): sampled
  samples (first and last included) bit-exact, plus count/argmax properties
  over all samples; hard_mnist_w4000 (batch 1024): every sample.
"""
import os

import numpy as np
import pytest
import torch

import oracle
import paper_2602_07400_gb300 as bl
from paper_2602_07400_gb300 import synth
from paper_2602_07400_gb300.pipeline import HardInfer, Network, TrainStep, unpack_bits
from parity_util import check_exact, check_fwd, check_grad

pytestmark = pytest.mark.gpu

oracle.set_threads(os.cpu_count() or 1)


def _step(wl, want_dx1, seed=0, k=None, keep_dy1=True, fuse_dy1=None, csr_order=True, node="soft", through=None,
          bytes1=None, bits1=None):
    if k is not None:
        wl = synth.Workload(wl.name, wl.batch, wl.d, wl.classes, wl.sigma, wl.thresholds, wl.widths, k, wl.tau)
    conn1, th1, conn2, th2 = synth.network(wl, seed)
    x, labels = synth.blob_batch(wl.batch, wl.d, wl.classes, wl.sigma, seed=seed + 7)
    net = Network(conn1, th1, conn2, th2, wl.w_in)
    st = TrainStep(net, wl.batch, wl.d, wl.thresholds, wl.classes, wl.tau, want_dx1=want_dx1,
                   keep_dy1=keep_dy1, fuse_dy1=fuse_dy1, csr_order=csr_order, node=node, through=through,
                   bytes1=bytes1, bits1=bits1)
    st.load(x.cuda(), labels.cuda())
    st.run()
    torch.cuda.synchronize()
    return wl, st, x.numpy(), labels.numpy(), (conn1, th1, conn2, th2)


def _check_grouped(st, dy2, wl):
    # the head's gradient rows: every node of a class shares its row
    g = wl.widths[1] // wl.classes
    rows = dy2.reshape(wl.classes, g, -1)
    assert np.all(rows == rows[:, :1, :])
    check_grad(st.dyg, rows[:, 0, :], "dY2 (per-class rows)")


def _full_compare(wl, st, x, labels, params, want_dx1, node="soft"):
    conn1, th1, conn2, th2 = params
    r = oracle.train_step(x, labels, wl.thresholds, conn1, th1, conn2, th2, wl.classes, wl.tau,
                          want_dx1=want_dx1, node=node)
    check_exact(st.wires().cpu().numpy().astype(np.float64), r["bits"], "bits")
    if node == "st":   # hard tables on binary inputs: every activation is a table entry
        check_exact(st.y1.cpu().numpy().astype(np.float64), r["y1"], "y1")
        check_exact(st.y2.cpu().numpy().astype(np.float64), r["y2"], "y2")
    check_fwd(st.y1, r["y1"], "y1")
    check_fwd(st.y2, r["y2"], "y2")
    check_fwd(st.logits, r["logits"], "logits")
    check_fwd(st.loss, np.array([r["loss"]]), "loss")
    _check_grouped(st, r["dy2"], wl)
    check_grad(st.dth2, r["dth2"], "dtheta2")
    check_grad(st.dy1, r["dy1"], "dy1")
    check_grad(st.dth1, r["dth1"], "dtheta1")
    if want_dx1:
        check_grad(st.dbits, r["dbits"], "dbits")


def test_tiny_step_all_outputs():
    wl, st, x, labels, params = _step(synth.WORKLOADS["tiny"], want_dx1=True)
    _full_compare(wl, st, x, labels, params, True)


@pytest.mark.parametrize("k,node", [(6, "soft"), (2, "soft"), (4, "soft"), (4, "st")])
def test_mnist_step_all_outputs(k, node):
    # k = 4 is the fan-in the paper pins for its comparisons (App. C.2)
    wl, st, x, labels, params = _step(synth.WORKLOADS["mnist"], want_dx1=False, k=k, node=node)
    _full_compare(wl, st, x, labels, params, False, node=node)


def test_tiny_step_st_all_outputs():
    # LightLUT straight-through: hard table samples forward, sigmoid-slope
    # dtheta, input gradients of the hard-table forward (both layers)
    wl, st, x, labels, params = _step(synth.WORKLOADS["tiny"], want_dx1=True, node="st")
    _full_compare(wl, st, x, labels, params, True, node="st")


@pytest.mark.parametrize("k", [6, 4])
def test_st_forward_is_the_deployed_network(k):
    # the straight-through forward of a batch equals the bit-packed hard
    # path on the discretized tables (App. C.1): layer-2 outputs bit for bit,
    # and head logits = popcounts / tau
    wl, st, x, labels, params = _step(synth.WORKLOADS["tiny"], want_dx1=False, k=k, node="st")
    hi = HardInfer(st.net, wl.batch, wl.d, wl.thresholds, wl.classes, keep_layer2=True)
    hi.x = st.x
    hi.binarize()
    hi.run()
    torch.cuda.synchronize()
    check_exact(st.y2.cpu().numpy().astype(np.uint8), unpack_bits(hi.yp2, wl.batch), "y2 vs hard layer 2")
    counts = hi.counts.cpu().numpy().astype(np.float64)
    check_fwd(st.logits, counts / wl.tau, "logits vs popcounts / tau")


@pytest.mark.parametrize("node", ["soft", "st"])
def test_mnist_k2_step_without_the_through_route(node):
    # k = 2 takes the through route by default (layer 1 recomputes its
    # output gradient through layer 2); the per-edge-term route still holds
    wl, st, x, labels, params = _step(synth.WORKLOADS["mnist"], want_dx1=False, k=2, node=node, through=False)
    assert not st.through
    _full_compare(wl, st, x, labels, params, False, node=node)


def test_mnist_k2_step_st_through():
    wl, st, x, labels, params = _step(synth.WORKLOADS["mnist"], want_dx1=False, k=2, node="st")
    assert st.through
    _full_compare(wl, st, x, labels, params, False, node="st")


@pytest.mark.parametrize("k,route", [(6, "fused"), (6, "csr"), (2, "through")])
def test_byte_wires_for_layer1_match_fp32_wires(k, route):
    # layer 1 on the encoder's wires as bytes (the step's default): the
    # forward is the table entry each sample selects, which the fp32 lerp tree
    # on the same wires reaches within the forward tolerance, and the table
    # gradient equals the fp32-row kernels' bit for bit given the same output
    # gradient: the dtheta-only kernel on dY1 (fused: layer 2's terms summed
    # inside the byte-row kernel; csr: the CSR reduction first), and the
    # through kernel on fp32 rows (k = 2)
    kw = {"fused": dict(fuse_dy1=True), "csr": dict(fuse_dy1=False), "through": {}}[route]
    wl, a, *_ = _step(synth.WORKLOADS["mnist"], want_dx1=False, k=k, bits1=False, **kw)
    assert a.bytes1 and a.bits.dtype == torch.uint8 and a.through == (route == "through")
    n = a.net
    bits32 = a.bits.float()
    y1 = torch.empty_like(a.y1)
    bl.bitlogic_lut_forward_node(bits32, n.conn1, n.theta1, y1)
    check_fwd(a.y1, y1.cpu().numpy().astype(np.float64), "y1 (lookup vs lerp tree)")
    ref = torch.empty_like(a.dth1)
    if route == "through":
        g = n.w2 // wl.classes
        bl.bitlogic_lut_backward_through(bits32, n.conn1, n.theta1, ref, a.y1, n.conn2, n.theta2, a.dyg, g,
                                         n.off2, n.edge2)
    else:
        bl.bitlogic_lut_backward_node(bits32, n.conn1, n.theta1, ref, "soft", dY=a.dy1)
    check_exact(a.dth1.cpu().numpy(), ref.cpu().numpy(), "dtheta1 (byte rows vs fp32 rows)")
    assert bl.bitlogic_device_error() == 0


@pytest.mark.parametrize("route", ["fused", "csr"])
def test_wire_bit_rows_equal_byte_wires(route):
    # the step's default off the through route: layer 1's wires at one bit
    # per sample; the lookup forward and the one-hot table gradient read the
    # same wires in the same order as the byte-row kernels, so every output
    # equals theirs bit for bit
    kw = dict(fuse_dy1=route == "fused")
    wl, a, *_ = _step(synth.WORKLOADS["mnist"], want_dx1=False, k=6, **kw)
    assert a.bits1 and a.bits.dtype == torch.int32 and a.bits.shape == (wl.w_in, bl.bitrow_words(wl.batch))
    _, b, *_ = _step(synth.WORKLOADS["mnist"], want_dx1=False, k=6, bits1=False, **kw)
    assert not b.bits1 and b.bits.dtype == torch.uint8
    check_exact(a.wires().cpu().numpy(), b.bits.cpu().numpy(), "wires")
    for name in ("y1", "y2", "logits", "loss", "dyg", "dy1", "dth1", "dth2"):
        check_exact(getattr(a, name).cpu().numpy(), getattr(b, name).cpu().numpy(), name)
    assert bl.bitlogic_device_error() == 0


def test_mnist_step_fused_layer1_gradient():
    # layer 1's output gradient summed inside its backward from layer 2's
    # CSR-ordered terms, instead of a CSR reduction followed by the
    # dtheta-only kernel
    wl, st, x, labels, params = _step(synth.WORKLOADS["mnist"], want_dx1=False, fuse_dy1=True)
    _full_compare(wl, st, x, labels, params, False)


def test_mnist_step_edge_ordered_terms():
    # layer 2's per-edge terms in edge order, read through the CSR edge map
    wl, st, x, labels, params = _step(synth.WORKLOADS["mnist"], want_dx1=False, csr_order=False)
    _full_compare(wl, st, x, labels, params, False)


def test_tiny_step_edge_ordered_terms():
    wl, st, x, labels, params = _step(synth.WORKLOADS["tiny"], want_dx1=True, csr_order=False)
    _full_compare(wl, st, x, labels, params, True)


@pytest.mark.parametrize("k", [6, 2])
def test_mnist_bench_configuration_matches(k):
    # the benchmark runs without storing dY1; its outputs equal the checked
    # configuration's bit for bit
    _, a, *_ = _step(synth.WORKLOADS["mnist"], want_dx1=False, keep_dy1=True, k=k)
    _, b, *_ = _step(synth.WORKLOADS["mnist"], want_dx1=False, keep_dy1=False, k=k)
    for name in ("y2", "logits", "loss", "dyg", "dth2", "dth1"):
        check_exact(getattr(b, name).cpu().numpy(), getattr(a, name).cpu().numpy(), name)


def test_graph_replay_matches_eager_launches():
    # the step captured once as CUDA graphs and replayed on new inputs gives
    # the eager launches' results bit for bit (training step and hard pass)
    wl = synth.WORKLOADS["tiny"]
    conn1, th1, conn2, th2 = synth.network(wl, 0)
    net = Network(conn1, th1, conn2, th2, wl.w_in)
    st = TrainStep(net, wl.batch, wl.d, wl.thresholds, wl.classes, wl.tau, want_dx1=True)
    hi = HardInfer(net, wl.batch, wl.d, wl.thresholds, wl.classes)
    hi.x = st.x
    x, labels = synth.blob_batch(wl.batch, wl.d, wl.classes, wl.sigma, seed=21)
    st.load(x.cuda(), labels.cuda())
    g_train, g_hard = st.capture(), hi.capture(binarize=True)
    x2, labels2 = synth.blob_batch(wl.batch, wl.d, wl.classes, wl.sigma, seed=22)
    st.load(x2.cuda(), labels2.cuda())
    g_train.replay()
    g_hard.replay()
    torch.cuda.synchronize()
    names = ("y1", "y2", "logits", "loss", "dyg", "dth1", "dth2", "dbits")
    got = {n: getattr(st, n).clone() for n in names}
    got_pred, got_counts = hi.pred.clone(), hi.counts.clone()
    st.run()
    hi.binarize()
    hi.run()
    torch.cuda.synchronize()
    for n in names:
        check_exact(got[n].cpu().numpy(), getattr(st, n).cpu().numpy(), n)
    check_exact(got_pred.cpu().numpy(), hi.pred.cpu().numpy(), "pred")
    check_exact(got_counts.cpu().numpy(), hi.counts.cpu().numpy(), "counts")
    # and the replayed step is the oracle's step on the new batch
    r = oracle.train_step(x2.numpy(), labels2.numpy(), wl.thresholds, conn1, th1, conn2, th2, wl.classes,
                          wl.tau, want_dx1=True)
    check_fwd(got["loss"], np.array([r["loss"]]), "loss")
    check_grad(got["dth1"], r["dth1"], "dtheta1")


def test_prefetcher_overlapped_steps_match_eager_steps():
    # batches streamed through the two-buffer prefetcher (copy of batch i+1
    # during step i) give every step's loss and predictions bit for bit
    from paper_2602_07400_gb300.pipeline import Prefetcher
    wl = synth.WORKLOADS["tiny"]
    conn1, th1, conn2, th2 = synth.network(wl, 0)
    net = Network(conn1, th1, conn2, th2, wl.w_in)
    st = TrainStep(net, wl.batch, wl.d, wl.thresholds, wl.classes, wl.tau)
    hi = HardInfer(net, wl.batch, wl.d, wl.thresholds, wl.classes)
    batches = [synth.blob_batch(wl.batch, wl.d, wl.classes, wl.sigma, seed=60 + i) for i in range(5)]
    want_loss, want_pred = [], []
    for x, labels in batches:
        st.load(x.cuda(), labels.cuda())
        st.run()
        hi.x.copy_(x.cuda())
        hi.binarize()
        hi.run()
        want_loss.append(float(st.loss.item()))
        want_pred.append(hi.pred.cpu().numpy().copy())
    hosts = [({"x": x.pin_memory(), "labels": l.pin_memory()}) for x, l in batches]
    pf = Prefetcher(st, ("x", "labels"), "loss")
    ph = Prefetcher(hi, ("x",), "pred", capture=lambda: hi.capture(binarize=True))
    loss_out = [torch.empty(1).pin_memory() for _ in batches]
    pred_out = [torch.empty(wl.batch, dtype=torch.int32).pin_memory() for _ in batches]
    pf.start()
    ph.start()
    pf.prefetch(hosts[0])
    ph.prefetch({"x": hosts[0]["x"]})
    for i in range(len(batches)):
        if i + 1 < len(batches):
            pf.prefetch(hosts[i + 1])
            ph.prefetch({"x": hosts[i + 1]["x"]})
        pf.run(loss_out[i])
        ph.run(pred_out[i])
    torch.cuda.synchronize()
    for i in range(len(batches)):
        assert float(loss_out[i][0]) == want_loss[i], i
        np.testing.assert_array_equal(pred_out[i].numpy(), want_pred[i])
    assert bl_device_ok()   # no run (the captures' warm-ups included) met a bad index or label


def _routed(wl, Kc, seed=0, node="soft"):
    from paper_2602_07400_gb300.pipeline import RoutedNetwork, RoutedTrainStep
    w1, w2 = wl.widths
    cand1 = synth.candidate_pools(w1 * wl.k, Kc, wl.w_in, seed)
    cand2 = synth.candidate_pools(w2 * wl.k, Kc, w1, seed + 1)
    r1 = synth.table_logits(w1 * wl.k, Kc, seed + 2, scale=0.5)
    r2 = synth.table_logits(w2 * wl.k, Kc, seed + 3, scale=0.5)
    th1 = synth.table_logits(w1, wl.K, seed + 100)
    th2 = synth.table_logits(w2, wl.K, seed + 101)
    net = RoutedNetwork(cand1, r1, th1, cand2, r2, th2, wl.w_in)
    st = RoutedTrainStep(net, wl.batch, wl.d, wl.thresholds, wl.classes, wl.tau, node=node)
    return net, st, (cand1, r1, th1, cand2, r2, th2)


@pytest.mark.parametrize("k,Kc,node", [(6, 8, "soft"), (4, 16, "soft"), (4, 16, "st")])
def test_tiny_routed_step_all_outputs(k, Kc, node):
    # learnable routing (candidate pools, softmax expected selection) in both
    # layers: every output and gradient, routing logits included
    wl = synth.WORKLOADS["tiny"]
    wl = synth.Workload(wl.name, wl.batch, wl.d, wl.classes, wl.sigma, wl.thresholds, wl.widths, k, wl.tau)
    net, st, (cand1, r1, th1, cand2, r2, th2) = _routed(wl, Kc)
    st.node = node
    x, labels = synth.blob_batch(wl.batch, wl.d, wl.classes, wl.sigma, seed=31)
    st.load(x.cuda(), labels.cuda())
    st.run()
    torch.cuda.synchronize()
    r = oracle.routed_train_step(x.numpy(), labels.numpy(), wl.thresholds, cand1, r1, th1, cand2, r2, th2,
                                 wl.classes, wl.tau, node=node)
    check_exact(st.bits.cpu().numpy().astype(np.float64), r["bits"], "bits")
    for name in ("xr1", "y1", "xr2", "y2", "logits"):
        check_fwd(getattr(st, name), r[name], name, atol=1e-6 if node == "st" else 0.0)
    check_fwd(st.loss, np.array([r["loss"]]), "loss")
    for name in ("dth2", "dr2", "dy1", "dth1", "dr1"):
        check_grad(getattr(st, name), r[name], name)
    check_grad(st.g2, r["dxr2"], "dXr2")
    assert bl_device_ok()


@pytest.mark.slow
def test_mnist_routed16_step_all_outputs():
    # the routed MNIST-shaped step at its benchmark size (8000 x 8000, k = 4,
    # 16 candidates per slot, batch 1024; layer 1 routed from byte wires),
    # routing logits drawn away from uniform so every softmax weight differs:
    # every output and gradient against the oracle
    wl = synth.WORKLOADS["mnist_k4_routed16"]
    net, st, (cand1, r1, th1, cand2, r2, th2) = _routed(wl, wl.Kc, seed=3)
    x, labels = synth.blob_batch(wl.batch, wl.d, wl.classes, wl.sigma, seed=41)
    st.load(x.cuda(), labels.cuda())
    st.run()
    torch.cuda.synchronize()
    r = oracle.routed_train_step(x.numpy(), labels.numpy(), wl.thresholds, cand1, r1, th1, cand2, r2, th2,
                                 wl.classes, wl.tau)
    check_exact(st.bits.cpu().numpy().astype(np.float64), r["bits"], "bits")
    for name in ("xr1", "y1", "xr2", "y2", "logits"):
        check_fwd(getattr(st, name), r[name], name)
    check_fwd(st.loss, np.array([r["loss"]]), "loss")
    for name in ("dth2", "dr2", "dy1", "dth1", "dr1"):
        check_grad(getattr(st, name), r[name], name)
    check_grad(st.g2, r["dxr2"], "dXr2")
    assert bl_device_ok()


def bl_device_ok():
    import paper_2602_07400_gb300 as bl
    return bl.bitlogic_device_error() == 0


def test_routed_training_learns_and_snaps_to_a_deployable_network():
    # AdamW on table and routing logits (routing logits start at zero, App. A);
    # the loss falls, and the snapped network's hard pass is the oracle's
    from paper_2602_07400_gb300.pipeline import RoutedNetwork, RoutedTrainStep
    wl = synth.WORKLOADS["tiny"]
    wl = synth.Workload(wl.name, wl.batch, wl.d, wl.classes, wl.sigma, wl.thresholds, wl.widths, 4, wl.tau)
    Kc = 8
    w1, w2 = wl.widths
    cand1 = synth.candidate_pools(w1 * 4, Kc, wl.w_in, 0)
    cand2 = synth.candidate_pools(w2 * 4, Kc, w1, 1)
    zeros1 = np.zeros((w1 * 4, Kc), np.float32)
    zeros2 = np.zeros((w2 * 4, Kc), np.float32)
    net = RoutedNetwork(cand1, zeros1, synth.table_logits(w1, 16, 100), cand2, zeros2,
                        synth.table_logits(w2, 16, 101), wl.w_in)
    st = RoutedTrainStep(net, wl.batch, wl.d, wl.thresholds, wl.classes, wl.tau)
    losses = []
    for step in range(1, 61):
        x, labels = synth.blob_batch(wl.batch, wl.d, wl.classes, wl.sigma, seed=200 + step, means_seed=7)
        st.load(x.cuda(), labels.cuda())
        st.run()
        st.update()
        losses.append(float(st.loss.item()))
    # uniform routing averages the pools at first, so the loss starts flat
    # and falls slowly at the paper's learning rate
    assert np.mean(losses[-5:]) < 0.97 * np.mean(losses[:3]), losses
    assert float(net.r1.abs().max()) > 0.0   # the routing logits moved
    fixed = net.snap()
    hi = HardInfer(fixed, 300, wl.d, wl.thresholds, wl.classes)
    x, _ = synth.blob_batch(300, wl.d, wl.classes, wl.sigma, seed=99)
    hi.x.copy_(x.cuda())
    hi.binarize()
    hi.run()
    torch.cuda.synchronize()
    conn1 = oracle.route_snap(cand1, net.r1.cpu().numpy()).reshape(w1, 4)
    conn2 = oracle.route_snap(cand2, net.r2.cpu().numpy()).reshape(w2, 4)
    t1 = oracle.binarize_tables(net.theta1.cpu().numpy())
    t2 = oracle.binarize_tables(net.theta2.cpu().numpy())
    ro = oracle.hard_infer(x.numpy(), wl.thresholds, conn1, t1, conn2, t2, wl.classes)
    check_exact(hi.counts.cpu().numpy(), ro["counts"], "counts of the snapped network")
    check_exact(hi.pred.cpu().numpy(), ro["pred"], "pred of the snapped network")


@pytest.mark.slow
def test_cifar10_step_all_outputs():
    # every element of every output and gradient of the CIFAR-10-shaped step
    # (64000 x 64000, B = 1024), against the oracle's full step
    wl, st, x, labels, params = _step(synth.WORKLOADS["cifar10"], want_dx1=False)
    _full_compare(wl, st, x, labels, params, False)


@pytest.mark.slow
def test_cifar100_step_all_outputs():
    # every element of every output and gradient of the CIFAR-100-shaped
    # step (128000 x 128000, B = 2048, 100 classes): about a minute and a half
    # of oracle time on 16 host cores
    wl, st, x, labels, params = _step(synth.WORKLOADS["cifar100"], want_dx1=False)
    _full_compare(wl, st, x, labels, params, False)


def _hard_run(wl, N, seed=0, samples=1536):
    conn1, th1, conn2, th2 = synth.network(wl, seed)
    net = Network(conn1, th1, conn2, th2, wl.w_in)
    hi = HardInfer(net, N, wl.d, wl.thresholds, wl.classes)
    x, labels = synth.blob_batch(N, wl.d, wl.classes, wl.sigma, seed=seed + 11, device="cuda")
    hi.x.copy_(x)
    del x, labels
    hi.binarize()
    hi.run()
    torch.cuda.synchronize()
    S = synth.sample_positions(N, samples, seed=seed)
    Sd = torch.from_numpy(S).cuda()
    xs = hi.x.index_select(0, Sd).cpu().numpy()
    t1 = oracle.binarize_tables(th1)
    t2 = oracle.binarize_tables(th2)
    check_exact(hi.table1.cpu().numpy().view(np.uint64), t1, "table1")
    check_exact(hi.table2.cpu().numpy().view(np.uint64), t2, "table2")
    r = oracle.hard_infer(xs, wl.thresholds, conn1, t1, conn2, t2, wl.classes)
    n = len(S)

    def cols(words):   # bits of the sampled samples, [rows, n]
        wsel = words.index_select(1, (Sd // 32)).cpu().numpy().view(np.uint32)
        return ((wsel >> (S % 32).astype(np.uint32)[None, :]) & 1).astype(np.uint8)

    check_exact(cols(hi.xp), unpack_bits(torch.from_numpy(r["xp"].view(np.int32)), n), "xp[sampled]")
    check_exact(cols(hi.yp1), unpack_bits(torch.from_numpy(r["yp1"].view(np.int32)), n), "yp1[sampled]")
    check_exact(hi.counts.index_select(0, Sd).cpu().numpy(), r["counts"], "counts[sampled]")
    check_exact(hi.pred.index_select(0, Sd).cpu().numpy(), r["pred"], "pred[sampled]")
    # properties over every sample: counts of a sample sum to the number of
    # ones among layer-2 outputs, each within [0, g]; pred is an argmax
    g = wl.widths[1] // wl.classes
    c = hi.counts
    assert int(c.min()) >= 0 and int(c.max()) <= g
    best = c.max(dim=1).values
    assert torch.equal(c.gather(1, hi.pred.long()[:, None])[:, 0], best)
    first = (c == best[:, None]).int().argmax(dim=1)
    assert torch.equal(first.int(), hi.pred)


def _hard_every_sample(wl, N, seed=0, chunk=1 << 16):
    """The hard pass on N samples on the GPU, then every sample recomputed by
    the oracle in chunks of `chunk` samples (a multiple of 32, so the chunks
    are whole packed words): the packed input, every layer-1 output word, the
    counts and the argmax of every sample, bit-exact."""
    assert chunk % 32 == 0
    conn1, th1, conn2, th2 = synth.network(wl, seed)
    net = Network(conn1, th1, conn2, th2, wl.w_in)
    hi = HardInfer(net, N, wl.d, wl.thresholds, wl.classes)
    x, labels = synth.blob_batch(N, wl.d, wl.classes, wl.sigma, seed=seed + 11, device="cuda")
    hi.x.copy_(x)
    del x, labels
    hi.binarize()
    hi.run()
    torch.cuda.synchronize()
    assert bl.bitlogic_device_error() == 0
    t1 = oracle.binarize_tables(th1)
    t2 = oracle.binarize_tables(th2)
    check_exact(hi.table1.cpu().numpy().view(np.uint64), t1, "table1")
    check_exact(hi.table2.cpu().numpy().view(np.uint64), t2, "table2")
    counts = hi.counts.cpu().numpy()
    pred = hi.pred.cpu().numpy()
    for s0 in range(0, N, chunk):
        s1 = min(N, s0 + chunk)
        w0, w1 = s0 // 32, (s1 + 31) // 32
        r = oracle.hard_infer(hi.x[s0:s1].cpu().numpy(), wl.thresholds, conn1, t1, conn2, t2, wl.classes)
        check_exact(hi.xp[:, w0:w1].cpu().numpy().view(np.uint32), r["xp"], f"xp words {w0}..{w1}")
        check_exact(hi.yp1[:, w0:w1].cpu().numpy().view(np.uint32), r["yp1"], f"yp1 words {w0}..{w1}")
        check_exact(counts[s0:s1], r["counts"], f"counts of samples {s0}..{s1}")
        check_exact(pred[s0:s1], r["pred"], f"pred of samples {s0}..{s1}")


@pytest.mark.slow
def test_hard_cifar10_every_sample():
    # the 2^22-sample hard pass of the CIFAR-10-shaped network: every sample
    # (packed input, layer-1 words, counts, argmax) against the oracle
    wl = synth.WORKLOADS["hard_cifar10"]
    _hard_every_sample(wl, wl.batch)


def test_hard_mnist_w4000_every_sample():
    # the deployed-MNIST shape (784 x 4 thresholds, 4000 x 4000, k = 4) at
    # batch 1024: every sample bit-exact against the oracle
    wl = synth.WORKLOADS["hard_mnist_w4000"]
    _hard_run(wl, wl.batch, samples=wl.batch)


@pytest.mark.slow
def test_hard_mnist_w4000_4m_sampled():
    wl = synth.WORKLOADS["hard_mnist_w4000_4m"]
    _hard_run(wl, wl.batch)


def test_hard_ragged_batch():
    wl = synth.WORKLOADS["hard_cifar10"]
    small = synth.Workload("hard_small", 0, wl.d, wl.classes, wl.sigma, wl.thresholds, (4000, 4000), 6, wl.tau)
    _hard_run(small, 100003, samples=700)
    _hard_run(small, 1024, samples=300)
    _hard_run(small, 37, samples=37)


def test_tiny_training_steps_match_oracle_and_lower_the_loss():
    # forward + backward + AdamW (§4 settings), repeated: the first two
    # updates of both layers' logits match the oracle's trajectory, and over
    # 30 steps on fresh batches of one dataset the loss falls
    wl = synth.WORKLOADS["tiny"]
    conn1, th1, conn2, th2 = synth.network(wl, 0)
    net = Network(conn1, th1, conn2, th2, wl.w_in)
    st = TrainStep(net, wl.batch, wl.d, wl.thresholds, wl.classes, wl.tau)
    o_th1, o_th2 = th1.astype(np.float64), th2.astype(np.float64)
    o_m = [np.zeros_like(o_th1), np.zeros_like(o_th2)]
    o_v = [np.zeros_like(o_th1), np.zeros_like(o_th2)]
    losses, accs = [], []
    for step in range(1, 31):
        x, labels = synth.blob_batch(wl.batch, wl.d, wl.classes, wl.sigma, seed=100 + step, means_seed=7)
        st.load(x.cuda(), labels.cuda())
        st.run()
        st.update()
        losses.append(float(st.loss.item()))
        accs.append(float((st.logits.argmax(1).cpu() == labels.long()).float().mean()))
        if step <= 2:
            # the oracle's step from the GPU's current logits, so each update
            # is checked on its own
            r = oracle.train_step(x.numpy(), labels.numpy(), wl.thresholds, conn1, o_th1.astype(np.float32),
                                  conn2, o_th2.astype(np.float32), wl.classes, wl.tau)
            o_th1, o_m[0], o_v[0] = oracle.adamw_step(o_th1, o_m[0], o_v[0], r["dth1"], step)
            o_th2, o_m[1], o_v[1] = oracle.adamw_step(o_th2, o_m[1], o_v[1], r["dth2"], step)
            # the step follows gradients held to 1e-4 relative: bound the
            # logits by 1e-5 relative plus 1e-3 of the learning rate
            for got, want, name in ((net.theta1, o_th1, "theta1"), (net.theta2, o_th2, "theta2")):
                err = np.abs(got.cpu().numpy().astype(np.float64) - want)
                assert np.all(err <= 1e-5 * np.abs(want) + 1e-3 * 0.01), f"{name} after step {step}: {err.max()}"
            o_th1 = net.theta1.cpu().numpy().astype(np.float64)
            o_th2 = net.theta2.cpu().numpy().astype(np.float64)
            o_m = [st.opt_m1.cpu().numpy().astype(np.float64), st.opt_m2.cpu().numpy().astype(np.float64)]
            o_v = [st.opt_v1.cpu().numpy().astype(np.float64), st.opt_v2.cpu().numpy().astype(np.float64)]
    # batches of one synthetic dataset (fixed class means): the loss falls and
    # the training accuracy climbs from chance
    assert np.mean(losses[-5:]) < 0.95 * np.mean(losses[:3]), losses
    assert accs[-1] >= 0.9, accs


def test_tiny_straight_through_training_lowers_the_loss():
    # the straight-through hard node trained with AdamW: its forward is the
    # deployed network at every step, and its loss still falls (30 steps)
    wl = synth.WORKLOADS["tiny"]
    conn1, th1, conn2, th2 = synth.network(wl, 0)
    net = Network(conn1, th1, conn2, th2, wl.w_in)
    st = TrainStep(net, wl.batch, wl.d, wl.thresholds, wl.classes, wl.tau, node="st")
    losses, accs = [], []
    for step in range(1, 31):
        x, labels = synth.blob_batch(wl.batch, wl.d, wl.classes, wl.sigma, seed=100 + step, means_seed=7)
        st.load(x.cuda(), labels.cuda())
        st.run()
        st.update()
        losses.append(float(st.loss.item()))
        accs.append(float((st.logits.argmax(1).cpu() == labels.long()).float().mean()))
        y2 = st.y2.cpu().numpy()
        assert np.all((y2 == 0.0) | (y2 == 1.0))
    assert np.mean(losses[-5:]) < 0.75 * np.mean(losses[:3]), losses
    assert accs[-1] >= 0.75, accs
