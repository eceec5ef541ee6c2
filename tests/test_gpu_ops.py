"""GPU-vs-oracle parity of each C-ABI call on small, ragged and degenerate
shapes (several tiles plus a tail), through the Python binding."""
import os

import numpy as np
import pytest
import torch

import oracle
import paper_2602_07400_gb300 as bl
from paper_2602_07400_gb300 import synth
from parity_util import check_exact, check_fwd, check_grad

pytestmark = pytest.mark.gpu

oracle.set_threads(os.cpu_count() or 1)


def dev(a, dtype=None):
    t = torch.from_numpy(np.ascontiguousarray(a))
    if dtype is not None:
        t = t.to(dtype)
    return t.cuda()


def no_device_error():
    assert bl.bitlogic_device_error() == 0


# ---------------------------------------------------------------- encoder --

@pytest.mark.parametrize("B,d,b", [(1, 5, 3), (37, 784, 3), (256, 70, 7), (1000, 33, 15), (65, 9, 32), (3, 1, 1),
                                   (1024, 784, 3), (132, 3072, 7)])
def test_encode_thermometer(B, d, b):
    rng = np.random.default_rng(B * 7 + d)
    x = rng.integers(0, 256, size=(B, d), dtype=np.uint8)
    thr = sorted(rng.choice(256, size=b, replace=False).tolist())
    bits = torch.full((d * b, B), -1.0, device="cuda")
    bl.bitlogic_encode_thermometer(dev(x), thr, bits)
    want = oracle.encode_thermometer(x, thr)
    check_exact(bits.cpu().numpy().astype(np.float64), want, "bits")
    # both forms in one pass: the same wires as fp32 rows and as byte rows
    bits2 = torch.full((d * b, B), -1.0, device="cuda")
    bits8 = torch.full((d * b, B), 7, dtype=torch.uint8, device="cuda")
    bl.bitlogic_encode_thermometer_both(dev(x), thr, bits2, bits8)
    check_exact(bits2.cpu().numpy().astype(np.float64), want, "bits (both)")
    check_exact(bits8.cpu().numpy().astype(np.float64), want, "bits8 (both)")
    no_device_error()


@pytest.mark.parametrize("B", [256, 255])
def test_encode_thermometer_edge_thresholds(B):
    # every byte value against the thresholds where the byte-wise test
    # changes form (T < 127: OR form, T >= 127: AND form, T = 255: nothing
    # exceeds it), on the vector (B % 4 == 0) and the scalar path
    d = 16
    x = ((np.arange(B * d, dtype=np.int64) * 37) % 256).astype(np.uint8).reshape(B, d)
    thr = [0, 1, 126, 127, 128, 254, 255]
    want = oracle.encode_thermometer(x, thr)
    bits = torch.full((d * len(thr), B), -1.0, device="cuda")
    bl.bitlogic_encode_thermometer(dev(x), thr, bits)
    check_exact(bits.cpu().numpy().astype(np.float64), want, "bits")
    bits8 = torch.full((d * len(thr), B), 7, dtype=torch.uint8, device="cuda")
    bl.bitlogic_encode_thermometer_u8(dev(x), thr, bits8)
    check_exact(bits8.cpu().numpy().astype(np.float64), want, "byte wires")
    no_device_error()


# ------------------------------------------------ quantile thermometer fit --

@pytest.mark.parametrize("n,offset,skew", [(1, 0, False), (15, 3, False), (16, 0, True), (17, 1, True),
                                           (4095, 7, False), (100003, 0, True), ((1 << 22) + 5, 9, True)])
def test_pixel_histogram_and_quantile_fit(n, offset, skew):
    rng = np.random.default_rng(n + offset)
    x = rng.integers(0, 256, size=n, dtype=np.uint8)
    if skew:   # a point mass at zero, as in digit images
        x[rng.random(n) < 0.85] = 0
    buf = torch.zeros(n + offset, dtype=torch.uint8, device="cuda")
    buf[offset:] = dev(x)
    view = buf[offset:]                        # offset bytes into the allocation
    hist = torch.zeros(256, dtype=torch.int64, device="cuda")
    bl.bitlogic_pixel_histogram(view, hist)
    want = np.bincount(x, minlength=256)
    check_exact(hist.cpu().numpy(), want, "histogram")
    bl.bitlogic_pixel_histogram(view, hist)   # counts accumulate
    check_exact(hist.cpu().numpy(), 2 * want, "histogram, two passes")
    for b in (1, 4, 8, 15, 32):
        got = bl.bitlogic_quantile_thresholds(hist, b)
        check_exact(got, oracle.quantile_thresholds(np.concatenate([x, x]), b), f"thresholds b={b}")


def test_quantile_fit_then_encode_mnist_shaped():
    # fit on several batches of the MNIST-shaped blobs, then encode with the
    # fitted thresholds (repeated ones included) through both encoders
    from paper_2602_07400_gb300.pipeline import fit_quantile_thresholds
    wl = synth.WORKLOADS["mnist"]
    xs = [synth.blob_batch(2048, wl.d, wl.classes, wl.sigma, seed=50 + i, means_seed=3)[0] for i in range(3)]
    for x in xs[:2]:
        x[:, : wl.d // 2] = 0                  # a third of all pixels black: the lowest thresholds repeat
    thr = fit_quantile_thresholds([x.cuda() for x in xs], 8)
    allx = np.concatenate([x.numpy() for x in xs])
    assert thr == [int(t) for t in oracle.quantile_thresholds(allx, 8)]
    assert thr[0] == thr[1] == 0
    x = xs[0][:300].numpy()
    bits = torch.empty(wl.d * 8, 300, device="cuda")
    bl.bitlogic_encode_thermometer(dev(x), thr, bits)
    check_exact(bits.cpu().numpy().astype(np.float64), oracle.encode_thermometer(x, thr), "bits")
    xp = torch.empty(wl.d * 8, (300 + 31) // 32, dtype=torch.int32, device="cuda")
    bl.bitlogic_pack_bits(dev(x), thr, xp)
    check_exact(xp.cpu().numpy().view(np.uint32), oracle.pack_bits(x, thr), "packed bits")


# ----------------------------------------------------------- soft forward --

SHAPES = [  # (k, w_in, w, B)
    (1, 3, 5, 1), (2, 7, 9, 5), (3, 40, 33, 37), (4, 100, 65, 128), (5, 64, 130, 259),
    (6, 300, 129, 256), (6, 6, 17, 100), (6, 1000, 64, 1027), (2, 2, 40, 64),
]


@pytest.mark.parametrize("k,w_in,w,B", SHAPES)
@pytest.mark.parametrize("binary", [False, True])
def test_lut_forward(k, w_in, w, B, binary):
    X = (synth.binary_activations if binary else synth.uniform_activations)(w_in, B, seed=k + B)
    conn = synth.connectivity(w, k, w_in, seed=w)
    theta = synth.table_logits(w, 1 << k, seed=k)
    Y = torch.full((w, B), np.nan, device="cuda")
    bl.bitlogic_lut_forward(dev(X), dev(conn), dev(theta), Y)
    check_fwd(Y, oracle.lut_forward(X.astype(np.float64), conn, theta), "Y")
    no_device_error()


def test_lut_forward_unaligned_scalar_path():
    # a view that starts 4 bytes into an allocation takes the scalar path
    k, w_in, w, B = 6, 50, 20, 64
    X = synth.uniform_activations(w_in, B, seed=1)
    conn = synth.connectivity(w, k, w_in, seed=2)
    theta = synth.table_logits(w, 64, seed=3)
    big = torch.zeros(w_in * B + 1, device="cuda")
    big[1:] = dev(X).reshape(-1)
    Xv = big[1:].view(w_in, B)
    Y = torch.empty(w, B, device="cuda")
    bl.bitlogic_lut_forward(Xv, dev(conn), dev(theta), Y)
    check_fwd(Y, oracle.lut_forward(X.astype(np.float64), conn, theta), "Y")


# ------------------------------------------- soft forward on byte rows --
#
# Binary wires as bytes: on binary inputs the corner weights are one-hot, so
# the layer returns the table entry each sample's input bits select (the
# oracle's multilinear form reaches it exactly on binary inputs).

@pytest.mark.parametrize("k,w_in,w,B", SHAPES)
@pytest.mark.parametrize("node", ["soft", "st"])
def test_lut_forward_u8(k, w_in, w, B, node):
    Xb = synth.binary_activations(w_in, B, seed=k + 3 * B)
    conn = synth.connectivity(w, k, w_in, seed=w + 7)
    theta = synth.table_logits(w, 1 << k, seed=k + 11)
    theta[0, :] = 0.0                    # ties sample 0 (st: [0 > 0] = 0)
    Y = torch.full((w, B), np.nan, device="cuda")
    bl.bitlogic_lut_forward_u8(dev(Xb.astype(np.uint8)), dev(conn), dev(theta), Y, node=node)
    want = oracle.lut_forward(Xb.astype(np.float64), conn, theta, node)
    if node == "st":
        check_exact(Y.cpu().numpy().astype(np.float64), want, "Y")
    else:
        check_fwd(Y, want, "Y")
    # the table entry itself: the sigmoid the fp32 kernels take, bit for bit
    idx = np.zeros((w, B), dtype=np.int64)
    for i in range(k):
        idx += Xb[conn[:, i]].astype(np.int64) << i
    tab = torch.sigmoid(dev(theta)).cpu().numpy() if node == "soft" else (theta > 0).astype(np.float32)
    entries = np.take_along_axis(tab, idx, axis=1)
    if node == "soft":
        check_fwd(Y, entries.astype(np.float64), "Y vs the selected entries")
    else:
        check_exact(Y.cpu().numpy(), entries, "Y vs the selected entries")
    no_device_error()


def test_lut_forward_u8_scalar_path_and_lowest_bit():
    # a view one byte into an allocation (and B % 4 != 0) takes the scalar
    # form; bytes other than 0 and 1 are read by their lowest bit
    k, w_in, w, B = 6, 50, 20, 67
    rng = np.random.default_rng(5)
    X = rng.integers(0, 256, size=(w_in, B), dtype=np.uint8)
    conn = synth.connectivity(w, k, w_in, seed=6)
    theta = synth.table_logits(w, 64, seed=7)
    big = torch.zeros(w_in * B + 1, dtype=torch.uint8, device="cuda")
    big[1:] = dev(X).reshape(-1)
    Y = torch.empty(w, B, device="cuda")
    bl.bitlogic_lut_forward_u8(big[1:].view(w_in, B), dev(conn), dev(theta), Y)
    check_fwd(Y, oracle.lut_forward((X & 1).astype(np.float64), conn, theta), "Y")
    for B2 in (64, 1024):   # the vector form with the same bytes
        X2 = rng.integers(0, 256, size=(w_in, B2), dtype=np.uint8)
        Y2 = torch.empty(w, B2, device="cuda")
        bl.bitlogic_lut_forward_u8(dev(X2), dev(conn), dev(theta), Y2)
        check_fwd(Y2, oracle.lut_forward((X2 & 1).astype(np.float64), conn, theta), "Y (vector)")
    no_device_error()


def test_lut_forward_u8_out_of_range_row_is_flagged():
    k, w_in, w, B = 3, 16, 8, 128
    Xb = synth.binary_activations(w_in, B, seed=9)
    conn = synth.connectivity(w, k, w_in, seed=10)
    conn[3, 1] = w_in + 5
    theta = synth.table_logits(w, 8, seed=11)
    assert bl.bitlogic_device_error() == 0
    Y = torch.empty(w, B, device="cuda")
    bl.bitlogic_lut_forward_u8(dev(Xb.astype(np.uint8)), dev(conn), dev(theta), Y)
    assert bl.bitlogic_device_error() == -8
    clamped = conn.copy()
    clamped[3, 1] = 0
    check_fwd(Y, oracle.lut_forward(Xb.astype(np.float64), clamped, theta), "Y (clamped)")


# ---------------------------------------------------------- soft backward --

@pytest.mark.parametrize("k,w_in,w,B", SHAPES)
def test_lut_backward(k, w_in, w, B):
    X = synth.uniform_activations(w_in, B, seed=k * 3 + B)
    conn = synth.connectivity(w, k, w_in, seed=w + 1)
    theta = synth.table_logits(w, 1 << k, seed=k + 5)
    dY = synth.uniform_gradients(w, B, seed=B, scale=1e-3)
    off, edge = bl.bitlogic_build_csr(conn, w_in)
    dth = torch.full((w, 1 << k), np.nan, device="cuda")
    dX = torch.full((w_in, B), np.nan, device="cuda")
    ws = torch.empty(bl.bitlogic_lut_backward_workspace(w_in, B, w, k, True), dtype=torch.uint8, device="cuda")
    bl.bitlogic_lut_backward(dev(X), dev(conn), dev(theta), dev(dY), dth, dX=dX,
                             csr_off=dev(off), csr_edge=dev(edge), workspace=ws)
    wth, wdx = oracle.lut_backward(X.astype(np.float64), conn, theta, dY.astype(np.float64))
    check_grad(dth, wth, "dtheta")
    check_grad(dX, wdx, "dX")
    # dX skipped: the dtheta-only kernel (another summation order), within
    # the tolerance of the oracle and deterministic from run to run
    dth2 = torch.full((w, 1 << k), np.nan, device="cuda")
    bl.bitlogic_lut_backward(dev(X), dev(conn), dev(theta), dev(dY), dth2)
    check_grad(dth2, wth, "dtheta without dX")
    dth3 = torch.full((w, 1 << k), np.nan, device="cuda")
    bl.bitlogic_lut_backward(dev(X), dev(conn), dev(theta), dev(dY), dth3)
    check_exact(dth3.cpu().numpy(), dth2.cpu().numpy(), "dtheta without dX, second run")
    no_device_error()


# ------------------------------------------ straight-through hard node --
#
# Forward and input gradient with the hard entries [theta > 0], dtheta with
# the sigmoid slope (LightLUT's straight-through form, §4 node sweep).

ST_ATOL = 1e-6   # fp32 evaluation of 0/1 tables on fractional inputs: absolute bound


@pytest.mark.parametrize("k,w_in,w,B", SHAPES)
@pytest.mark.parametrize("binary", [False, True])
def test_lut_forward_st(k, w_in, w, B, binary):
    X = (synth.binary_activations if binary else synth.uniform_activations)(w_in, B, seed=k + 2 * B)
    conn = synth.connectivity(w, k, w_in, seed=w + 3)
    theta = synth.table_logits(w, 1 << k, seed=k + 9)
    theta[0, :] = 0.0                    # ties sample 0
    Y = torch.full((w, B), np.nan, device="cuda")
    bl.bitlogic_lut_forward_node(dev(X), dev(conn), dev(theta), Y, node="st")
    want = oracle.lut_forward(X.astype(np.float64), conn, theta, "st")
    if binary:   # integer arithmetic in fp32: the deployed table entries exactly
        check_exact(Y.cpu().numpy().astype(np.float64), want, "Y")
    else:
        check_fwd(Y, want, "Y", atol=ST_ATOL)
    no_device_error()


@pytest.mark.parametrize("k,w_in,w,B", SHAPES)
@pytest.mark.parametrize("binary", [False, True])
def test_lut_backward_st(k, w_in, w, B, binary):
    X = (synth.binary_activations if binary else synth.uniform_activations)(w_in, B, seed=k * 5 + B)
    conn = synth.connectivity(w, k, w_in, seed=w + 4)
    theta = synth.table_logits(w, 1 << k, seed=k + 11)
    dY = synth.uniform_gradients(w, B, seed=B + 1, scale=1e-3)
    off, edge = bl.bitlogic_build_csr(conn, w_in)
    dth = torch.full((w, 1 << k), np.nan, device="cuda")
    P = torch.full((w * k, B), np.nan, device="cuda")
    bl.bitlogic_lut_backward_node(dev(X), dev(conn), dev(theta), dth, node="st", dY=dev(dY), edge_terms=P)
    dX = torch.full((w_in, B), np.nan, device="cuda")
    bl.bitlogic_csr_reduce(P, dev(off), dev(edge), dX)
    wth, wdx = oracle.lut_backward(X.astype(np.float64), conn, theta, dY.astype(np.float64), node="st")
    check_grad(dth, wth, "dtheta")
    check_grad(dX, wdx, "dX")
    # the soft node on the same inputs gives the same dtheta (the estimator
    # keeps the sigmoid slope) but another dX
    wth_s, _ = oracle.lut_backward(X.astype(np.float64), conn, theta, dY.astype(np.float64), want_dx=False)
    np.testing.assert_allclose(wth, wth_s, rtol=1e-12, atol=0)
    # without dX: the dtheta-only kernel serves both forms
    dth2 = torch.full((w, 1 << k), np.nan, device="cuda")
    bl.bitlogic_lut_backward_node(dev(X), dev(conn), dev(theta), dth2, node="st", dY=dev(dY))
    check_grad(dth2, wth, "dtheta without dX")
    no_device_error()


# ------------------------------------------------------ learnable routing --

ROUTE = [  # (slots, Kc, w_in, B)
    (1, 1, 1, 1), (5, 3, 7, 37), (24, 4, 50, 128), (64, 8, 300, 259), (96, 16, 1000, 1024),
    (40, 32, 64, 100), (33, 16, 2352, 1027), (7, 5, 9, 4),
]


@pytest.mark.parametrize("slots,Kc,w_in,B", ROUTE)
def test_route_forward_backward(slots, Kc, w_in, B):
    rng = np.random.default_rng(slots * 31 + Kc)
    X = synth.uniform_activations(w_in, B, seed=slots + B)
    cand = synth.candidate_pools(slots, Kc, w_in, seed=Kc + 3)
    r = synth.table_logits(slots, Kc, seed=slots + 4)
    G = synth.uniform_gradients(slots, B, seed=B + 5, scale=1e-3)
    Xr = torch.full((slots, B), np.nan, device="cuda")
    prob = torch.full((slots, Kc), np.nan, device="cuda")
    bl.bitlogic_route_forward(dev(X), dev(cand), dev(r), Xr, prob)
    wXr, wp = oracle.route_forward(X.astype(np.float64), cand, r)
    check_fwd(Xr, wXr, "Xr")
    check_fwd(prob, wp, "prob")
    off, edge = bl.bitlogic_build_csr(cand, w_in)
    dr = torch.full((slots, Kc), np.nan, device="cuda")
    dX = torch.full((w_in, B), np.nan, device="cuda")
    bl.bitlogic_route_backward(dev(X), dev(cand), dev(r), dev(G), dr, prob, dev(off), dev(edge), dX)
    wdr, wdX = oracle.route_backward(X.astype(np.float64), cand, r, G.astype(np.float64))
    check_grad(dr, wdr, "dr")
    check_grad(dX, wdX, "dX")
    dr2 = torch.full((slots, Kc), np.nan, device="cuda")
    bl.bitlogic_route_backward(dev(X), dev(cand), dev(r), dev(G), dr2)   # dr only
    check_exact(dr2.cpu().numpy(), dr.cpu().numpy(), "dr without dX")
    conn = torch.full((slots,), -1, dtype=torch.int32, device="cuda")
    bl.bitlogic_route_snap(dev(cand), dev(r), conn)
    check_exact(conn.cpu().numpy(), oracle.route_snap(cand, r), "snap")
    no_device_error()


@pytest.mark.parametrize("slots,Kc,w_in,B,binary", [(96, 16, 2352, 1024, True), (33, 8, 300, 259, True),
                                                     (40, 32, 64, 100, False), (7, 5, 9, 4, False)])
def test_route_over_byte_rows(slots, Kc, w_in, B, binary):
    # routing over a uint8 layer input (the encoder's 0/1 wires, or any bytes)
    # against the oracle on the same values
    rng = np.random.default_rng(slots + Kc)
    X8 = (rng.integers(0, 2, size=(w_in, B)) if binary else rng.integers(0, 256, size=(w_in, B))).astype(np.uint8)
    cand = synth.candidate_pools(slots, Kc, w_in, seed=Kc)
    r = synth.table_logits(slots, Kc, seed=slots)
    G = synth.uniform_gradients(slots, B, seed=B, scale=1e-3)
    Xr = torch.full((slots, B), np.nan, device="cuda")
    prob = torch.empty(slots, Kc, device="cuda")
    bl.bitlogic_route_forward_u8(dev(X8), dev(cand), dev(r), Xr, prob)
    wXr, wp = oracle.route_forward(X8.astype(np.float64), cand, r)
    check_fwd(Xr, wXr, "Xr from bytes")
    check_fwd(prob, wp, "prob")
    dr = torch.full((slots, Kc), np.nan, device="cuda")
    bl.bitlogic_route_backward_u8(dev(X8), dev(cand), dev(r), dev(G), dr)
    wdr, _ = oracle.route_backward(X8.astype(np.float64), cand, r, G.astype(np.float64), want_dx=False)
    check_grad(dr, wdr, "dr from bytes")
    # equal to the fp32 calls on the same values bit for bit (the same
    # products in the same order)
    Xf = dev(X8.astype(np.float32))
    Xr_f = torch.empty_like(Xr)
    bl.bitlogic_route_forward(Xf, dev(cand), dev(r), Xr_f)
    check_exact(Xr.cpu().numpy(), Xr_f.cpu().numpy(), "Xr bytes vs fp32")
    dr_f = torch.empty_like(dr)
    bl.bitlogic_route_backward(Xf, dev(cand), dev(r), dev(G), dr_f)
    check_exact(dr.cpu().numpy(), dr_f.cpu().numpy(), "dr bytes vs fp32")
    no_device_error()


@pytest.mark.parametrize("B,d,b", [(1, 5, 3), (37, 784, 3), (256, 70, 7), (1024, 784, 4)])
def test_encode_thermometer_bytes(B, d, b):
    rng = np.random.default_rng(B + d)
    x = rng.integers(0, 256, size=(B, d), dtype=np.uint8)
    thr = sorted(rng.choice(256, size=b, replace=False).tolist())
    bits = torch.full((d * b, B), 7, dtype=torch.uint8, device="cuda")
    bl.bitlogic_encode_thermometer_u8(dev(x), thr, bits)
    check_exact(bits.cpu().numpy().astype(np.float64), oracle.encode_thermometer(x, thr), "byte wires")


def test_route_unaligned_and_tied_logits():
    # a view 4 bytes into an allocation takes the scalar paths; tied logits
    # snap to the first candidate
    slots, Kc, w_in, B = 12, 8, 40, 64
    X = synth.uniform_activations(w_in, B, seed=1)
    cand = synth.candidate_pools(slots, Kc, w_in, seed=2)
    r = np.zeros((slots, Kc), np.float32)
    r[:, 3] = 1.0
    r[:, 6] = 1.0
    big = torch.zeros(w_in * B + 1, device="cuda")
    big[1:] = dev(X).reshape(-1)
    Xv = big[1:].view(w_in, B)
    Xr = torch.empty(slots, B, device="cuda")
    bl.bitlogic_route_forward(Xv, dev(cand), dev(r), Xr)
    check_fwd(Xr, oracle.route_forward(X.astype(np.float64), cand, r)[0], "Xr (scalar path)")
    G = synth.uniform_gradients(slots, B, seed=3, scale=1e-3)
    dr = torch.empty(slots, Kc, device="cuda")
    bl.bitlogic_route_backward(Xv, dev(cand), dev(r), dev(G), dr)
    check_grad(dr, oracle.route_backward(X.astype(np.float64), cand, r, G.astype(np.float64), False)[0], "dr")
    conn = torch.empty(slots, dtype=torch.int32, device="cuda")
    bl.bitlogic_route_snap(dev(cand), dev(r), conn)
    check_exact(conn.cpu().numpy(), cand[:, 3], "snap to the first maximum")


@pytest.mark.parametrize("k,w_in,w,B,group", [(6, 300, 120, 256, 12), (6, 64, 40, 1024, 40), (3, 50, 30, 37, 5),
                                               (2, 9, 20, 100, 1), (1, 4, 6, 8, 3)])
def test_backward_grouped_dy(k, w_in, w, B, group):
    # dY given as one row per group of `group` consecutive nodes
    X = synth.uniform_activations(w_in, B, seed=k + B)
    conn = synth.connectivity(w, k, w_in, seed=w)
    theta = synth.table_logits(w, 1 << k, seed=k)
    rows = synth.uniform_gradients(w // group, B, seed=group, scale=1e-3)
    dY = np.repeat(rows, group, axis=0)
    dth = torch.empty(w, 1 << k, device="cuda")
    P = torch.empty(w * k, B, device="cuda")
    out = torch.empty(w, B, device="cuda")
    bl.bitlogic_lut_backward_ex(dev(X), dev(conn), dev(theta), dth, dY=dev(rows), dy_group=group,
                                edge_terms=P, dY_out=out)
    check_exact(out.cpu().numpy(), dY, "dY_out")
    off, edge = bl.bitlogic_build_csr(conn, w_in)
    dX = torch.empty(w_in, B, device="cuda")
    bl.bitlogic_csr_reduce(P, dev(off), dev(edge), dX)
    wth, wdx = oracle.lut_backward(X.astype(np.float64), conn, theta, dY.astype(np.float64))
    check_grad(dth, wth, "dtheta")
    check_grad(dX, wdx, "dX")
    # same as the ungrouped call on the expanded dY, bit for bit
    dth2 = torch.empty(w, 1 << k, device="cuda")
    P2 = torch.empty(w * k, B, device="cuda")
    bl.bitlogic_lut_backward_edges(dev(X), dev(conn), dev(theta), dev(dY), dth2, P2)
    check_exact(dth2.cpu().numpy(), dth.cpu().numpy(), "dtheta grouped vs full")
    check_exact(P2.cpu().numpy(), P.cpu().numpy(), "edge terms grouped vs full")


@pytest.mark.parametrize("k,w_in,w,B", [(6, 200, 150, 256), (6, 1000, 300, 1024), (4, 40, 64, 36),
                                        (2, 12, 30, 7), (1, 5, 8, 64)])
def test_backward_from_upstream_terms(k, w_in, w, B):
    # layer A (this call) gets its output gradient as the CSR sum of layer
    # B's per-edge terms; equals csr_reduce + backward_edges bit for bit
    kb, wb = 3, 2 * w
    X = synth.uniform_activations(w_in, B, seed=B)
    conn = synth.connectivity(w, k, w_in, seed=1)
    theta = synth.table_logits(w, 1 << k, seed=2)
    conn_b = synth.connectivity(wb, kb, w, seed=3)       # layer B reads layer A's outputs
    off_b, edge_b = bl.bitlogic_build_csr(conn_b, w)
    terms = synth.uniform_gradients(wb * kb, B, seed=4, scale=1e-3)
    dth = torch.empty(w, 1 << k, device="cuda")
    out = torch.empty(w, B, device="cuda")
    P = torch.empty(w * k, B, device="cuda")
    bl.bitlogic_lut_backward_ex(dev(X), dev(conn), dev(theta), dth, up_terms=dev(terms),
                                up_off=dev(off_b), up_edge=dev(edge_b), edge_terms=P, dY_out=out)
    dY_ref = torch.empty(w, B, device="cuda")
    bl.bitlogic_csr_reduce(dev(terms), dev(off_b), dev(edge_b), dY_ref)
    check_exact(out.cpu().numpy(), dY_ref.cpu().numpy(), "dY from terms vs csr_reduce")
    dth_ref = torch.empty(w, 1 << k, device="cuda")
    P_ref = torch.empty(w * k, B, device="cuda")
    bl.bitlogic_lut_backward_edges(dev(X), dev(conn), dev(theta), dY_ref, dth_ref, P_ref)
    check_exact(dth.cpu().numpy(), dth_ref.cpu().numpy(), "dtheta fused vs unfused")
    check_exact(P.cpu().numpy(), P_ref.cpu().numpy(), "edge terms fused vs unfused")
    # and against the oracle on the dense dY of the upstream terms
    dY = np.zeros((w, B))
    for e in range(wb * kb):
        dY[conn_b.reshape(-1)[e]] += terms[e].astype(np.float64)
    wth, _ = oracle.lut_backward(X.astype(np.float64), conn, theta, dY, want_dx=False)
    check_grad(dth, wth, "dtheta")
    # without this layer's own terms: the dtheta-only kernel reads the
    # upstream rows through its ring (another summation order for dtheta)
    dth_t = torch.full((w, 1 << k), np.nan, device="cuda")
    out_t = torch.full((w, B), np.nan, device="cuda")
    bl.bitlogic_lut_backward_ex(dev(X), dev(conn), dev(theta), dth_t, up_terms=dev(terms),
                                up_off=dev(off_b), up_edge=dev(edge_b), dY_out=out_t)
    check_exact(out_t.cpu().numpy(), out.cpu().numpy(), "dY from terms (dtheta-only kernel)")
    check_grad(dth_t, wth, "dtheta (dtheta-only kernel)")
    # the same with every per-edge buffer in CSR order: upstream rows
    # permuted to CSR positions (no edge map), this layer's terms stored at
    # its own CSR positions; all results identical bit for bit
    off_a, edge_a = bl.bitlogic_build_csr(conn, w_in)
    pos_a = bl.bitlogic_csr_positions(edge_a)
    dth_c = torch.empty(w, 1 << k, device="cuda")
    out_c = torch.empty(w, B, device="cuda")
    P_c = torch.full((w * k, B), np.nan, device="cuda")
    bl.bitlogic_lut_backward_ex(dev(X), dev(conn), dev(theta), dth_c, up_terms=dev(terms[edge_b]),
                                up_off=dev(off_b), up_edge=None, edge_terms=P_c, edge_pos=dev(pos_a),
                                dY_out=out_c)
    check_exact(out_c.cpu().numpy(), out.cpu().numpy(), "dY from CSR-ordered terms")
    check_exact(dth_c.cpu().numpy(), dth.cpu().numpy(), "dtheta from CSR-ordered terms")
    check_exact(P_c.cpu().numpy(), P.cpu().numpy()[edge_a], "edge terms stored in CSR order")
    dX = torch.empty(w_in, B, device="cuda")
    dX_c = torch.empty(w_in, B, device="cuda")
    bl.bitlogic_csr_reduce(P, dev(off_a), dev(edge_a), dX)
    bl.bitlogic_csr_reduce(P_c, dev(off_a), None, dX_c)
    check_exact(dX_c.cpu().numpy(), dX.cpu().numpy(), "csr_reduce of CSR-ordered terms")
    no_device_error()
    no_device_error()


def test_backward_is_deterministic_and_handles_skewed_consumers():
    # 3 inputs shared by 500 nodes (fan-in 2): every input has ~333 consumers
    k, w_in, w, B = 2, 3, 500, 96
    X = synth.uniform_activations(w_in, B, seed=1)
    conn = synth.connectivity(w, k, w_in, seed=2)
    theta = synth.table_logits(w, 4, seed=3)
    dY = synth.uniform_gradients(w, B, seed=4, scale=1e-2)
    off, edge = bl.bitlogic_build_csr(conn, w_in)
    ws = torch.empty(bl.bitlogic_lut_backward_workspace(w_in, B, w, k, True), dtype=torch.uint8, device="cuda")
    outs = []
    for _ in range(2):
        dth = torch.empty(w, 4, device="cuda")
        dX = torch.empty(w_in, B, device="cuda")
        bl.bitlogic_lut_backward(dev(X), dev(conn), dev(theta), dev(dY), dth, dX=dX,
                                 csr_off=dev(off), csr_edge=dev(edge), workspace=ws)
        outs.append((dth.cpu().numpy(), dX.cpu().numpy()))
    check_exact(outs[0][0], outs[1][0], "dtheta run-to-run")
    check_exact(outs[0][1], outs[1][1], "dX run-to-run")
    wth, wdx = oracle.lut_backward(X.astype(np.float64), conn, theta, dY.astype(np.float64))
    check_grad(outs[0][0], wth, "dtheta")
    check_grad(outs[0][1], wdx, "dX")


THROUGH = [  # (k, ku, w_in, w, up_w, up_group, B)
    (2, 2, 50, 64, 80, 8, 128), (6, 2, 300, 200, 150, 1, 260), (3, 3, 40, 96, 120, 12, 4),
    (2, 1, 30, 40, 60, 6, 1028), (4, 3, 100, 256, 512, 64, 132), (1, 2, 9, 12, 20, 20, 8),
]


def _through_oracle(X, conn, theta, Y, up_conn, up_theta, up_dY, up_group, node):
    # the next layer's per-node output gradient rows, its input gradient by
    # the oracle's scatter-add, then this layer's table gradient
    dY2 = np.repeat(np.asarray(up_dY, np.float64), up_group, axis=0)
    _, g = oracle.lut_backward(Y, up_conn, up_theta, dY2, want_dx=True, node=node)
    dth, _ = oracle.lut_backward(X, conn, theta, g, want_dx=False, node=node)
    return dth, g


@pytest.mark.parametrize("node", ["soft", "st"])
@pytest.mark.parametrize("k,ku,w_in,w,up_w,up_group,B", THROUGH)
def test_lut_backward_through(k, ku, w_in, w, up_w, up_group, B, node):
    # this layer's table gradient with its output gradient recomputed through
    # the next layer, against the oracle's two-layer chain rule
    X = synth.uniform_activations(w_in, B, seed=k + 10)
    conn = synth.connectivity(w, k, w_in, seed=k + 11)
    theta = synth.table_logits(w, 1 << k, seed=k + 12)
    Y = synth.uniform_activations(w, B, seed=k + 13)
    up_conn = synth.connectivity(up_w, ku, w, seed=ku + 14)
    up_theta = synth.table_logits(up_w, 1 << ku, seed=ku + 15)
    up_dY = synth.uniform_gradients(up_w // up_group, B, seed=16, scale=1e-3)
    off, edge = bl.bitlogic_build_csr(up_conn, w)
    dth = torch.full((w, 1 << k), np.nan, device="cuda")
    g = torch.full((w, B), np.nan, device="cuda")
    bl.bitlogic_lut_backward_through(dev(X), dev(conn), dev(theta), dth, dev(Y), dev(up_conn), dev(up_theta),
                                     dev(up_dY), up_group, dev(off), dev(edge), node=node, dY_out=g)
    wdth, wg = _through_oracle(X, conn, theta, Y, up_conn, up_theta, up_dY, up_group, node)
    check_grad(g, wg, "dY (recomputed)")
    check_grad(dth, wdth, "dtheta")
    # without the optional output: the same table gradient bit for bit
    dth2 = torch.empty_like(dth)
    bl.bitlogic_lut_backward_through(dev(X), dev(conn), dev(theta), dth2, dev(Y), dev(up_conn), dev(up_theta),
                                     dev(up_dY), up_group, dev(off), dev(edge), node=node)
    check_exact(dth2.cpu().numpy(), dth.cpu().numpy(), "dtheta without dY_out")
    no_device_error()


def test_lut_backward_through_many_and_no_consumers():
    # inputs with more than 32 consumers (the consumer list is taken in
    # chunks of 32) and inputs nobody reads (zero output gradient)
    k, ku, w_in, w, up_w, B = 2, 2, 20, 40, 300, 64
    rng = np.random.default_rng(3)
    up_conn = np.stack([rng.choice([0, 1, 2, 3, 5], size=2, replace=False) for _ in range(up_w)]).astype(np.int32)
    X = synth.uniform_activations(w_in, B, seed=1)
    conn = synth.connectivity(w, k, w_in, seed=2)
    theta = synth.table_logits(w, 4, seed=3)
    Y = synth.uniform_activations(w, B, seed=4)
    up_theta = synth.table_logits(up_w, 4, seed=5)
    up_dY = synth.uniform_gradients(up_w, B, seed=6)
    off, edge = bl.bitlogic_build_csr(up_conn, w)
    assert np.diff(off).max() > 64
    dth = torch.empty(w, 4, device="cuda")
    g = torch.full((w, B), np.nan, device="cuda")
    bl.bitlogic_lut_backward_through(dev(X), dev(conn), dev(theta), dth, dev(Y), dev(up_conn), dev(up_theta),
                                     dev(up_dY), 1, dev(off), dev(edge), dY_out=g)
    wdth, wg = _through_oracle(X, conn, theta, Y, up_conn, up_theta, up_dY, 1, "soft")
    check_grad(g, wg, "dY (recomputed)")
    check_grad(dth, wdth, "dtheta")
    unused = np.setdiff1d(np.arange(w), up_conn.reshape(-1))
    assert unused.size > 0
    assert torch.all(g[torch.from_numpy(unused).cuda()] == 0)
    no_device_error()


def test_lut_backward_through_identity_edge_map():
    # up_edge = NULL: the next layer's edges already in CSR order (node j2
    # reads inputs 2 j2 and 2 j2 + 1, so edge e feeds input e)
    k, ku, w_in, w, B = 3, 2, 30, 64, 256
    up_w = w // 2
    up_conn = np.arange(w, dtype=np.int32).reshape(up_w, 2)
    X = synth.uniform_activations(w_in, B, seed=1)
    conn = synth.connectivity(w, k, w_in, seed=2)
    theta = synth.table_logits(w, 8, seed=3)
    Y = synth.uniform_activations(w, B, seed=4)
    up_theta = synth.table_logits(up_w, 4, seed=5)
    up_dY = synth.uniform_gradients(up_w, B, seed=6)
    off, edge = bl.bitlogic_build_csr(up_conn, w)
    assert np.array_equal(edge, np.arange(w))
    dth = torch.empty(w, 8, device="cuda")
    bl.bitlogic_lut_backward_through(dev(X), dev(conn), dev(theta), dth, dev(Y), dev(up_conn), dev(up_theta),
                                     dev(up_dY), 1, dev(off), None)
    wdth, _ = _through_oracle(X, conn, theta, Y, up_conn, up_theta, up_dY, 1, "soft")
    check_grad(dth, wdth, "dtheta")
    no_device_error()


BYTES = [(1, 10, 7, 4), (2, 50, 64, 128), (3, 40, 33, 260), (4, 100, 65, 1028), (5, 64, 40, 132),
         (6, 300, 129, 1024), (6, 2000, 77, 516)]


@pytest.mark.parametrize("node", ["soft", "st"])
@pytest.mark.parametrize("k,w_in,w,B", BYTES)
def test_lut_backward_u8_rows_and_terms(k, w_in, w, B, node):
    # byte-row input (binary wires): dtheta from dY rows and from the next
    # layer's per-edge terms, equal bit for bit to the fp32-row dtheta-only
    # backward on the same wires (the terms summed by bitlogic_csr_reduce
    # first), and within the parity tolerance of the oracle
    Xb = synth.binary_activations(w_in, B, seed=k + 20)
    X8 = dev(Xb.astype(np.uint8))
    conn = synth.connectivity(w, k, w_in, seed=k + 21)
    theta = synth.table_logits(w, 1 << k, seed=k + 22)
    dY = synth.uniform_gradients(w, B, seed=k + 23, scale=1e-3)
    ref = torch.empty(w, 1 << k, device="cuda")
    bl.bitlogic_lut_backward_node(dev(Xb), dev(conn), dev(theta), ref, node, dY=dev(dY))
    got = torch.full((w, 1 << k), np.nan, device="cuda")
    out = torch.full((w, B), np.nan, device="cuda")
    bl.bitlogic_lut_backward_u8(X8, dev(conn), dev(theta), got, node, dY=dev(dY), dY_out=out)
    check_exact(got.cpu().numpy(), ref.cpu().numpy(), "dtheta (rows) vs fp32 rows")
    check_exact(out.cpu().numpy(), dY, "dY_out (rows)")
    wdth, _ = oracle.lut_backward(Xb, conn, theta, dY, want_dx=False, node=node)
    check_grad(got, wdth, "dtheta (rows) vs oracle")
    # per-edge terms of a next layer (fan-in 3 over these w rows), in CSR order
    up_w = max(4, w // 2)
    up_conn = synth.connectivity(up_w, 3, w, seed=k + 24)
    off, edge = bl.bitlogic_build_csr(up_conn, w)
    terms = synth.uniform_gradients(up_w * 3, B, seed=k + 25, scale=1e-3)
    summed = torch.empty(w, B, device="cuda")
    bl.bitlogic_csr_reduce(dev(terms), dev(off), dev(edge), summed)
    ref2 = torch.empty(w, 1 << k, device="cuda")
    bl.bitlogic_lut_backward_node(dev(Xb), dev(conn), dev(theta), ref2, node, dY=summed)
    got2 = torch.full((w, 1 << k), np.nan, device="cuda")
    out2 = torch.full((w, B), np.nan, device="cuda")
    bl.bitlogic_lut_backward_u8(X8, dev(conn), dev(theta), got2, node, up_terms=dev(terms), up_off=dev(off),
                                up_edge=dev(edge), dY_out=out2)
    check_exact(out2.cpu().numpy(), summed.cpu().numpy(), "dY_out (terms) vs CSR reduction")
    check_exact(got2.cpu().numpy(), ref2.cpu().numpy(), "dtheta (terms) vs fp32 rows")
    no_device_error()


@pytest.mark.parametrize("k,group", [(6, 4), (3, 13), (2, 52)])
def test_lut_backward_u8_grouped_rows(k, group):
    # dY rows shared by groups of nodes (the head's per-class rows): the
    # byte-row kernel equals the fp32-row dtheta-only kernel bit for bit
    w_in, w, B = 90, 52, 516
    Xb = synth.binary_activations(w_in, B, seed=k + 60)
    conn = synth.connectivity(w, k, w_in, seed=k + 61)
    theta = synth.table_logits(w, 1 << k, seed=k + 62)
    dY = synth.uniform_gradients(w // group, B, seed=k + 63, scale=1e-3)
    ref = torch.empty(w, 1 << k, device="cuda")
    bl.bitlogic_lut_backward_node(dev(Xb), dev(conn), dev(theta), ref, "soft", dY=dev(dY), dy_group=group)
    got = torch.full((w, 1 << k), np.nan, device="cuda")
    bl.bitlogic_lut_backward_u8(dev(Xb.astype(np.uint8)), dev(conn), dev(theta), got, dY=dev(dY), dy_group=group)
    check_exact(got.cpu().numpy(), ref.cpu().numpy(), "dtheta (grouped rows)")
    dYfull = np.repeat(dY, group, axis=0)
    wdth, _ = oracle.lut_backward(Xb, conn, theta, dYfull, want_dx=False)
    check_grad(got, wdth, "dtheta (grouped rows) vs oracle")
    no_device_error()


@pytest.mark.parametrize("k", [2, 6])
def test_lut_backward_u8_terms_with_many_and_no_consumers(k):
    # the term rows of a node beyond the ones its ring slot holds (ten), and
    # beyond 32 (read in chunks), and nodes with no consumers: the same sum
    # as the CSR reduction, bit for bit, and the same dtheta as the fp32
    # dtheta-only kernel on it
    w_in, w, up_w, B = 50, 40, 300, 260
    rng = np.random.default_rng(7)
    up_conn = np.stack([rng.choice([0, 1, 2, 3, 5, 8, 13], size=2, replace=False)
                        for _ in range(up_w)]).astype(np.int32)
    up_conn[:12] = np.arange(14, 38, dtype=np.int32).reshape(12, 2)   # 24 rows with one consumer
    up_conn[12:41] = [9, 10]                                            # two rows with 29
    off, edge = bl.bitlogic_build_csr(up_conn, w)
    deg = np.diff(off)
    assert (deg > 32).any() and ((deg > 10) & (deg <= 32)).any() and (deg == 0).any() and (deg == 1).any()
    Xb = synth.binary_activations(w_in, B, seed=k + 30)
    conn = synth.connectivity(w, k, w_in, seed=k + 31)
    theta = synth.table_logits(w, 1 << k, seed=k + 32)
    terms = synth.uniform_gradients(up_w * 2, B, seed=k + 33, scale=1e-3)
    summed = torch.empty(w, B, device="cuda")
    bl.bitlogic_csr_reduce(dev(terms), dev(off), dev(edge), summed)
    ref = torch.empty(w, 1 << k, device="cuda")
    bl.bitlogic_lut_backward_node(dev(Xb), dev(conn), dev(theta), ref, dY=summed)
    got = torch.full((w, 1 << k), np.nan, device="cuda")
    out = torch.full((w, B), np.nan, device="cuda")
    bl.bitlogic_lut_backward_u8(dev(Xb.astype(np.uint8)), dev(conn), dev(theta), got, up_terms=dev(terms),
                                up_off=dev(off), up_edge=dev(edge), dY_out=out)
    check_exact(out.cpu().numpy(), summed.cpu().numpy(), "dY_out vs CSR reduction")
    check_exact(got.cpu().numpy(), ref.cpu().numpy(), "dtheta vs fp32 rows")
    wdth, _ = oracle.lut_backward(Xb, conn, theta, summed.cpu().numpy().astype(np.float64), want_dx=False)
    check_grad(got, wdth, "dtheta vs oracle")
    assert torch.all(out[torch.from_numpy(np.nonzero(deg == 0)[0]).cuda()] == 0)
    no_device_error()


def test_lut_backward_through_u8_equals_fp32():
    k, ku, w_in, w, up_w, up_group, B = 6, 2, 300, 200, 150, 5, 260
    Xb = synth.binary_activations(w_in, B, seed=1)
    conn = synth.connectivity(w, k, w_in, seed=2)
    theta = synth.table_logits(w, 1 << k, seed=3)
    Y = synth.uniform_activations(w, B, seed=4)
    up_conn = synth.connectivity(up_w, ku, w, seed=5)
    up_theta = synth.table_logits(up_w, 1 << ku, seed=6)
    up_dY = synth.uniform_gradients(up_w // up_group, B, seed=7, scale=1e-3)
    off, edge = bl.bitlogic_build_csr(up_conn, w)
    a = torch.empty(w, 1 << k, device="cuda")
    b = torch.empty(w, 1 << k, device="cuda")
    args = (dev(Y), dev(up_conn), dev(up_theta), dev(up_dY), up_group, dev(off), dev(edge))
    bl.bitlogic_lut_backward_through(dev(Xb), dev(conn), dev(theta), a, *args)
    bl.bitlogic_lut_backward_through_u8(dev(Xb.astype(np.uint8)), dev(conn), dev(theta), b, *args)
    check_exact(b.cpu().numpy(), a.cpu().numpy(), "through dtheta, byte rows vs fp32 rows")
    no_device_error()


def test_backward_unused_inputs_get_zero():
    k, w_in, w, B = 3, 50, 4, 40     # at most 12 of 50 inputs are read
    X = synth.uniform_activations(w_in, B, seed=5)
    conn = synth.connectivity(w, k, w_in, seed=6)
    theta = synth.table_logits(w, 8, seed=7)
    dY = synth.uniform_gradients(w, B, seed=8)
    off, edge = bl.bitlogic_build_csr(conn, w_in)
    dX = torch.full((w_in, B), np.nan, device="cuda")
    ws = torch.empty(bl.bitlogic_lut_backward_workspace(w_in, B, w, k, True), dtype=torch.uint8, device="cuda")
    bl.bitlogic_lut_backward(dev(X), dev(conn), dev(theta), dev(dY), torch.empty(w, 8, device="cuda"),
                             dX=dX, csr_off=dev(off), csr_edge=dev(edge), workspace=ws)
    unused = np.setdiff1d(np.arange(w_in), conn.reshape(-1))
    assert unused.size > 0
    assert torch.all(dX[torch.from_numpy(unused).cuda()] == 0)


def test_empty_batch_is_a_noop():
    k, w_in, w = 2, 5, 3
    conn = dev(synth.connectivity(w, k, w_in, seed=1))
    theta = dev(synth.table_logits(w, 4, seed=1))
    X = torch.empty(w_in, 0, device="cuda")
    Y = torch.empty(w, 0, device="cuda")
    bl.bitlogic_lut_forward(X, conn, theta, Y)
    dth = torch.full((w, 4), 7.0, device="cuda")
    bl.bitlogic_lut_backward(X, conn, theta, torch.empty(w, 0, device="cuda"), dth)
    assert torch.all(dth == 0)
    xp = torch.empty(10, 0, dtype=torch.int32, device="cuda")
    bl.bitlogic_pack_bits(torch.empty(0, 5, dtype=torch.uint8, device="cuda"), [1, 2], xp)
    # straight-through node, routing: an empty batch leaves the batch sums at
    # zero, and the routing forward still gives the slot probabilities
    dth = torch.full((w, 4), 7.0, device="cuda")
    bl.bitlogic_lut_backward_node(X, conn, theta, dth, node="st", dY=torch.empty(w, 0, device="cuda"))
    assert torch.all(dth == 0)
    slots, Kc = 6, 3
    cand = synth.candidate_pools(slots, Kc, w_in, seed=2)
    r = synth.table_logits(slots, Kc, seed=3)
    prob = torch.full((slots, Kc), np.nan, device="cuda")
    bl.bitlogic_route_forward(X, dev(cand), dev(r), torch.empty(slots, 0, device="cuda"), prob)
    check_fwd(prob, oracle.route_forward(np.zeros((w_in, 1)), cand, r)[1], "prob of an empty batch")
    dr = torch.full((slots, Kc), 7.0, device="cuda")
    bl.bitlogic_route_backward(X, dev(cand), dev(r), torch.empty(slots, 0, device="cuda"), dr)
    assert torch.all(dr == 0)
    hist = torch.zeros(256, dtype=torch.int64, device="cuda")
    bl.bitlogic_pixel_histogram(torch.empty(0, dtype=torch.uint8, device="cuda"), hist)
    assert int(hist.sum()) == 0
    no_device_error()


# -------------------------------------------------------------------- head --

@pytest.mark.parametrize("C,g,B,tau", [(10, 100, 256, 10.0), (3, 7, 37, 2.0), (100, 13, 259, 100.0),
                                       (1, 40, 5, 1.0), (10, 800, 1, 20.0),
                                       (3, 1025, 256, 5.0), (10, 6400, 256, 50.0)])   # rows split over blocks
def test_head_loss(C, g, B, tau):
    rng = np.random.default_rng(C + B)
    Y = rng.random((C * g, B)).astype(np.float32)
    labels = rng.integers(0, C, size=B).astype(np.int32)
    loss = torch.zeros(1, device="cuda")
    logits = torch.empty(B, C, device="cuda")
    dY = torch.empty(C * g, B, device="cuda")
    ws = torch.empty(bl.bitlogic_head_loss_workspace(B, C), dtype=torch.uint8, device="cuda")
    bl.bitlogic_head_loss(dev(Y), dev(labels), C, tau, loss, ws, logits=logits, dY=dY)
    wl, wloss, wdy = oracle.head_loss(Y.astype(np.float64), labels, C, tau)
    check_fwd(logits, wl, "logits")
    check_fwd(loss, np.array([wloss]), "loss")
    check_grad(dY, wdy, "dY")
    # optional outputs absent
    loss2 = torch.zeros(1, device="cuda")
    bl.bitlogic_head_loss(dev(Y), dev(labels), C, tau, loss2, ws)
    check_exact(loss2.cpu().numpy(), loss.cpu().numpy(), "loss without optional outputs")
    no_device_error()


def test_head_grouped_gradient_rows():
    C, g, B = 10, 80, 259
    rng = np.random.default_rng(3)
    Y = rng.random((C * g, B)).astype(np.float32)
    labels = rng.integers(0, C, size=B).astype(np.int32)
    ws = torch.empty(bl.bitlogic_head_loss_workspace(B, C), dtype=torch.uint8, device="cuda")
    dY = torch.empty(C * g, B, device="cuda")
    dYg = torch.empty(C, B, device="cuda")
    loss = torch.zeros(1, device="cuda")
    bl.bitlogic_head_loss_ex(dev(Y), dev(labels), C, 7.0, loss, ws, dY=dY, dY_grouped=dYg)
    full = dY.cpu().numpy().reshape(C, g, B)
    for c in range(C):
        check_exact(full[c], np.repeat(dYg[c:c + 1].cpu().numpy(), g, axis=0), f"class {c}")


# -------------------------------------------------------------------- hard --

def test_binarize_tables():
    rng = np.random.default_rng(3)
    for k in (1, 2, 5, 6):
        theta = rng.standard_normal((77, 1 << k)).astype(np.float32)
        theta[::5, 0] = 0.0
        theta[1::7, -1] = -0.0
        theta[2::9, 0] = np.float32(1e-45)
        tab = torch.empty(77, dtype=torch.int64, device="cuda")
        bl.bitlogic_binarize_tables(dev(theta), tab)
        check_exact(tab.cpu().numpy().view(np.uint64), oracle.binarize_tables(theta), f"table k={k}")


@pytest.mark.parametrize("N,d,b", [(1, 5, 3), (31, 8, 1), (32, 16, 7), (33, 9, 3), (1000, 784, 3),
                                   (1025, 24, 15), (5000, 3, 32), (70000, 17, 2)])
def test_pack_bits(N, d, b):
    rng = np.random.default_rng(N + d)
    x = rng.integers(0, 256, size=(N, d), dtype=np.uint8)
    thr = sorted(rng.choice(256, size=b, replace=False).tolist())
    xp = torch.full((d * b, (N + 31) // 32), -1, dtype=torch.int32, device="cuda")
    bl.bitlogic_pack_bits(dev(x), thr, xp)
    check_exact(xp.cpu().numpy().view(np.uint32), oracle.pack_bits(x, thr), "xp")


HARD = [  # (k, w_in, w, N)
    (1, 3, 5, 1), (2, 10, 9, 31), (3, 40, 33, 33), (4, 100, 65, 1000), (5, 64, 100, 1025),
    (6, 300, 129, 4096), (6, 7, 20, 70001), (6, 2000, 256, 100000),
    (6, 16384, 300, 32891),   # staged path over two word chunks (768 + 260 words)
]


@pytest.mark.parametrize("k,w_in,w,N", HARD)
def test_hard_forward(k, w_in, w, N):
    W = (N + 31) // 32
    xp = synth.random_words(w_in, W, seed=N)
    if N % 32:
        xp[:, -1] &= np.uint32((1 << (N % 32)) - 1)
    conn = synth.connectivity(w, k, w_in, seed=k)
    table = synth.random_tables(w, seed=w)
    if k < 6:
        table &= np.uint64((1 << (1 << k)) - 1)
    yp = torch.full((w, W), -1, dtype=torch.int32, device="cuda")
    bl.bitlogic_hard_forward(dev(xp.view(np.int32)), N, dev(conn), dev(table.view(np.int64)), yp=yp)
    check_exact(yp.cpu().numpy().view(np.uint32), oracle.hard_forward(xp, N, conn, table), "yp")
    no_device_error()


@pytest.mark.parametrize("k,w_in,C,g,N", [(6, 200, 10, 100, 1024), (6, 300, 3, 7, 37), (4, 50, 10, 33, 5000),
                                          (2, 9, 1, 13, 100), (6, 500, 10, 1500, 70001), (6, 64, 2, 9000, 999)])
def test_hard_forward_popcount_head(k, w_in, C, g, N):
    w = C * g
    W = (N + 31) // 32
    xp = synth.random_words(w_in, W, seed=N + 1)
    if N % 32:
        xp[:, -1] &= np.uint32((1 << (N % 32)) - 1)
    conn = synth.connectivity(w, k, w_in, seed=k + 1)
    table = synth.random_tables(w, seed=w + 1)
    counts = torch.full((N, C), -1, dtype=torch.int32, device="cuda")
    pred = torch.full((N,), -1, dtype=torch.int32, device="cuda")
    yp = torch.full((w, W), -1, dtype=torch.int32, device="cuda")
    bl.bitlogic_hard_forward(dev(xp.view(np.int32)), N, dev(conn), dev(table.view(np.int64)),
                             yp=yp, C=C, counts=counts, pred=pred)
    wyp = oracle.hard_forward(xp, N, conn, table)
    wc, wp = oracle.popcount_head(wyp, N, C)
    check_exact(yp.cpu().numpy().view(np.uint32), wyp, "yp")
    check_exact(counts.cpu().numpy(), wc, "counts")
    check_exact(pred.cpu().numpy(), wp, "pred")
    # head without yp and pred
    counts2 = torch.full((N, C), -1, dtype=torch.int32, device="cuda")
    bl.bitlogic_hard_forward(dev(xp.view(np.int32)), N, dev(conn), dev(table.view(np.int64)),
                             C=C, counts=counts2)
    check_exact(counts2.cpu().numpy(), wc, "counts (no yp)")


def test_hard_equals_soft_on_binarized_tables():
    # the correctness anchor of App. C.1 on the GPU: the soft kernel on binary
    # inputs with theta = +-800 (t exactly 0 or 1) equals the hard kernel
    k, w_in, w, N = 6, 200, 96, 256
    rng = np.random.default_rng(1)
    Xb = rng.integers(0, 2, size=(w_in, N)).astype(np.float32)
    conn = synth.connectivity(w, k, w_in, seed=1)
    theta = synth.table_logits(w, 64, seed=2)
    th_hard = np.where(theta > 0, 800.0, -800.0).astype(np.float32)
    Y = torch.empty(w, N, device="cuda")
    bl.bitlogic_lut_forward(dev(Xb), dev(conn), dev(th_hard), Y)
    W = N // 32
    xp = np.zeros((w_in, W), np.uint32)
    for s in range(N):
        xp[:, s // 32] |= Xb[:, s].astype(np.uint32) << np.uint32(s % 32)
    tab = torch.empty(w, dtype=torch.int64, device="cuda")
    bl.bitlogic_binarize_tables(dev(theta), tab)
    yp = torch.empty(w, W, dtype=torch.int32, device="cuda")
    bl.bitlogic_hard_forward(dev(xp.view(np.int32)), N, dev(conn), tab, yp=yp)
    from paper_2602_07400_gb300.pipeline import unpack_bits
    check_exact(Y.cpu().numpy(), unpack_bits(yp, N).astype(np.float32), "soft vs hard")


# -------------------------------------------------------- error handling --

def test_out_of_range_connectivity_is_flagged_not_faulted():
    # an index past w_in reaches the kernel (bypassing the host CSR check):
    # the kernel reads row 0 instead and raises the device flag
    k, w_in, w, B = 2, 10, 4, 32
    conn = synth.connectivity(w, k, w_in, seed=1)
    bad = conn.copy()
    bad[2, 1] = w_in + 5
    theta = synth.table_logits(w, 4, seed=1)
    X = synth.uniform_activations(w_in, B, seed=1)
    assert bl.bitlogic_device_error() == 0
    Y = torch.empty(w, B, device="cuda")
    bl.bitlogic_lut_forward(dev(X), dev(bad), dev(theta), Y)
    assert bl.bitlogic_device_error() == -8
    assert bl.bitlogic_device_error() == 0          # the flag was cleared
    clamped = bad.copy()
    clamped[2, 1] = 0
    check_fwd(Y, oracle.lut_forward(X.astype(np.float64), clamped, theta), "Y (clamped)")
    yp = torch.empty(w, 1, dtype=torch.int32, device="cuda")
    bl.bitlogic_hard_forward(torch.zeros(w_in, 1, dtype=torch.int32, device="cuda"), 32,
                             dev(bad), torch.zeros(w, dtype=torch.int64, device="cuda"), yp=yp)
    assert bl.bitlogic_device_error() == -8


def test_bad_label_is_flagged():
    C, g, B = 3, 4, 8
    Y = torch.rand(C * g, B, device="cuda")
    labels = torch.tensor([0, 1, 2, 3, 0, 1, 2, 0], dtype=torch.int32, device="cuda")
    ws = torch.empty(bl.bitlogic_head_loss_workspace(B, C), dtype=torch.uint8, device="cuda")
    bl.bitlogic_head_loss(Y, labels, C, 1.0, torch.zeros(1, device="cuda"), ws)
    assert bl.bitlogic_device_error() == -8


def test_binding_rejects_wrong_tensors():
    X = torch.rand(10, 8, device="cuda")
    conn = torch.zeros(4, 2, dtype=torch.int32, device="cuda")
    theta = torch.zeros(4, 4, device="cuda")
    with pytest.raises(TypeError):
        bl.bitlogic_lut_forward(X.double(), conn, theta, torch.empty(4, 8, device="cuda"))
    with pytest.raises(ValueError):
        bl.bitlogic_lut_forward(X, conn, theta, torch.empty(4, 9, device="cuda"))
    with pytest.raises(ValueError):
        bl.bitlogic_lut_forward(X.cpu(), conn, theta, torch.empty(4, 8, device="cuda"))


def test_issue_probe_runs_every_kind():
    # the throughput probe behind the pipe rates the benchmark reports: every
    # thread writes the combination of its chains, every block (one per SM)
    # its clock cycles, which grow with the iteration count
    n = bl.bitlogic_issue_probe_threads()
    nb = bl.bitlogic_issue_probe_blocks()
    assert n == 1024 * nb
    sink = torch.zeros(n, dtype=torch.int32, device="cuda")
    cyc = torch.zeros(nb, dtype=torch.int64, device="cuda")
    for kind in ("lop3", "imad", "ffma", "mux3", "mix"):
        sink.zero_()
        bl.bitlogic_issue_probe(kind, 4, sink, cyc, seed=12345)
        torch.cuda.synchronize()
        assert int((sink != 0).sum()) > n // 2, kind
        short = cyc.clone()
        bl.bitlogic_issue_probe(kind, 64, sink, cyc, seed=12345)
        torch.cuda.synchronize()
        assert bool((short > 0).all()) and bool((cyc > short).all()), kind
    bl.bitlogic_issue_probe("mix", 4, sink)   # cycles are optional
    with pytest.raises(ValueError):
        bl.bitlogic_issue_probe("lop4", 1, sink)
    with pytest.raises(bl.BitLogicError):
        bl.bitlogic_issue_probe(7, 1, sink)


# ------------------------------------------------------------------ AdamW --

@pytest.mark.parametrize("n,wd", [(4096, 0.0), (1000003, 0.0), (64000 * 64, 0.1), (7, 0.05)])
def test_adamw_update(n, wd):
    # two steps in a row (steps 1 and 2, the state carried on the device),
    # each against the oracle from the same inputs; the error scale of each
    # moment update is the size of its two terms
    rng = np.random.default_rng(n)
    theta = rng.standard_normal(n).astype(np.float32)
    m = np.zeros(n, np.float32)
    v = np.zeros(n, np.float32)
    th_d, m_d, v_d = dev(theta), dev(m), dev(v)
    for step in (1, 2):
        g = (rng.standard_normal(n) * 10.0 ** rng.integers(-7, -1, size=n)).astype(np.float32)
        g[::97] = 0.0
        bl.bitlogic_adamw_update(th_d, m_d, v_d, dev(g), step, lr=0.01, weight_decay=wd)
        # the oracle gets the hyperparameters as the kernel receives them (fp32)
        f = lambda a: float(np.float32(a))
        th_o, m_o, v_o = oracle.adamw_step(theta, m, v, g, step, lr=f(0.01), beta1=f(0.9), beta2=f(0.999),
                                           eps=f(1e-8), wd=f(wd))
        got_th, got_m, got_v = (t.cpu().numpy().astype(np.float64) for t in (th_d, m_d, v_d))
        scale_m = 0.9 * np.abs(m) + 0.1 * np.abs(g.astype(np.float64))
        scale_v = 0.999 * np.abs(v) + 0.001 * g.astype(np.float64) ** 2
        # theta: the step is at most a few learning rates, so its terms are
        # |theta| and 4 lr (a result near 0 comes from cancellation)
        scale_th = np.abs(theta.astype(np.float64)) + 4 * 0.01
        assert np.all(np.abs(got_m - m_o) <= 1e-6 * scale_m + 1e-30), "m"
        assert np.all(np.abs(got_v - v_o) <= 1e-6 * scale_v + 1e-30), "v"
        err = np.abs(got_th - th_o)
        assert np.all(err <= 1e-6 * scale_th), f"theta: {err.max()}"
        theta, m, v = got_th.astype(np.float32), got_m.astype(np.float32), got_v.astype(np.float32)
    no_device_error()
