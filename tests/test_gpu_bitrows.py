"""GPU parity of layer 1 on wire bit rows (binary wires at one bit per
sample): the encoder against the oracle's thermometer, and the lookup
forward and one-hot table gradient against the byte-row kernels on the same
wires (bit for bit) and against the oracle.  The host-side packing below
writes the documented layout (bit 8m + r of word L of a 1024-sample block is
sample 128r + 4L + m) so that any binary rows can be fed in."""
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

# thresholds on both sides of the byte-wise test's two forms and at its edges
EDGE_THR = [0, 1, 126, 127, 128, 200, 254, 255]


def dev(a):
    return torch.from_numpy(np.ascontiguousarray(a)).cuda()


def pack_rows(X):
    """Binary rows [w, B] (0/1) to wire bit rows [w, bitrow_words(B)] int32."""
    w, B = X.shape
    nblk = (B + 1023) // 1024
    P = np.zeros((w, nblk * 1024), dtype=np.uint64)
    P[:, :B] = X.astype(np.uint64) & 1
    P = P.reshape(w, nblk, 8, 32, 4)               # [row, block, r, L, m]
    shift = (8 * np.arange(4)[None, None, None, None, :] + np.arange(8)[None, None, :, None, None])
    words = (P << shift.astype(np.uint64)).sum(axis=(2, 4))   # [row, block, L]
    return words.reshape(w, nblk * 32).astype(np.uint32).view(np.int32)


def unpack_rows(words, B):
    w = words.shape[0]
    u = words.view(np.uint32).reshape(w, -1, 1, 32, 1).astype(np.uint64)
    shift = (8 * np.arange(4)[None, None, None, None, :] + np.arange(8)[None, None, :, None, None])
    bits = (u >> shift.astype(np.uint64)) & 1                  # [row, block, r, L, m]
    return bits.reshape(w, -1)[:, :B].astype(np.uint8)


def test_pack_rows_layout():
    # the layout written out: sample 128 r + 4 L + m of block q at bit 8 m + r
    # of word 32 q + L
    B = 2048 + 12
    X = np.zeros((1, B), np.uint8)
    for s in (0, 1, 5, 130, 1023, 1024, 2047, 2048 + 11):
        X[0, s] = 1
    W = pack_rows(X).view(np.uint32)
    assert W.shape == (1, bl.bitrow_words(B)) == (1, 96)
    for s in np.nonzero(X[0])[0]:
        q, o = divmod(int(s), 1024)
        r, rem = divmod(o, 128)
        L, m = divmod(rem, 4)
        assert (W[0, 32 * q + L] >> (8 * m + r)) & 1
    assert int(sum(bin(int(v)).count("1") for v in W[0])) == 8
    np.testing.assert_array_equal(unpack_rows(W.view(np.int32), B), X)


@pytest.mark.parametrize("B,d,b", [(4, 1, 1), (1000, 8, 8), (1024, 784, 3), (1028, 33, 15), (2048, 3072, 15),
                                   (3, 17, 32), (4100, 16, 8)])
def test_encode_thermometer_bitrows(B, d, b):
    rng = np.random.default_rng(B + d)
    x = rng.integers(0, 256, size=(B, d), dtype=np.uint8)
    x[:, 0] = np.arange(B) % 256
    thr = list(EDGE_THR) if b == len(EDGE_THR) else sorted(rng.integers(0, 256, size=b).tolist())
    words = torch.full((d * b, bl.bitrow_words(B)), -1, dtype=torch.int32, device="cuda")
    bl.bitlogic_encode_thermometer_bitrows(dev(x), thr, words)
    want = oracle.encode_thermometer(x, thr)
    got = words.cpu().numpy()
    check_exact(unpack_rows(got, B).astype(np.float64), want, "wires")
    np.testing.assert_array_equal(got, pack_rows(want.astype(np.uint8)))   # samples past B read 0
    # a sample matrix one byte into an allocation (the byte-load form)
    big = torch.zeros(B * d + 1, dtype=torch.uint8, device="cuda")
    big[1:] = dev(x).reshape(-1)
    words2 = torch.full_like(words, -1)
    bl.bitlogic_encode_thermometer_bitrows(big[1:].view(B, d), thr, words2)
    np.testing.assert_array_equal(words2.cpu().numpy(), got)


FWD = [(1, 10, 7, 4), (2, 50, 64, 128), (3, 40, 33, 260), (4, 100, 65, 1028), (5, 64, 40, 132),
       (6, 300, 129, 1024), (6, 2000, 77, 2052), (6, 90, 40, 67), (3, 20, 9, 1)]


@pytest.mark.parametrize("node", ["soft", "st"])
@pytest.mark.parametrize("k,w_in,w,B", FWD)
def test_lut_forward_bitrows(k, w_in, w, B, node):
    Xb = synth.binary_activations(w_in, B, seed=k + 3 * B)
    conn = synth.connectivity(w, k, w_in, seed=w + 7)
    theta = synth.table_logits(w, 1 << k, seed=k + 11)
    theta[0, :] = 0.0
    Y = torch.full((w, B), np.nan, device="cuda")
    bl.bitlogic_lut_forward_bitrows(dev(pack_rows(Xb)), B, dev(conn), dev(theta), Y, node=node)
    ref = torch.full((w, B), np.nan, device="cuda")
    bl.bitlogic_lut_forward_u8(dev(Xb.astype(np.uint8)), dev(conn), dev(theta), ref, node=node)
    check_exact(Y.cpu().numpy(), ref.cpu().numpy(), "Y vs byte rows")
    want = oracle.lut_forward(Xb.astype(np.float64), conn, theta, node)
    if node == "st":
        check_exact(Y.cpu().numpy().astype(np.float64), want, "Y vs oracle")
    else:
        check_fwd(Y, want, "Y vs oracle")
    assert bl.bitlogic_device_error() == 0


def test_lut_forward_bitrows_out_of_range_row_is_flagged():
    k, w_in, w, B = 3, 16, 8, 1100
    Xb = synth.binary_activations(w_in, B, seed=9)
    conn = synth.connectivity(w, k, w_in, seed=10)
    conn[3, 1] = w_in + 5
    theta = synth.table_logits(w, 8, seed=11)
    assert bl.bitlogic_device_error() == 0
    Y = torch.empty(w, B, device="cuda")
    bl.bitlogic_lut_forward_bitrows(dev(pack_rows(Xb)), B, dev(conn), dev(theta), Y)
    assert bl.bitlogic_device_error() == -8
    clamped = conn.copy()
    clamped[3, 1] = 0
    check_fwd(Y, oracle.lut_forward(Xb.astype(np.float64), clamped, theta), "Y (clamped)")


BWD = [(1, 10, 7, 4), (2, 50, 64, 128), (3, 40, 33, 260), (4, 100, 65, 1028), (5, 64, 40, 132),
       (6, 300, 129, 1024), (6, 2000, 77, 2052)]


@pytest.mark.parametrize("node", ["soft", "st"])
@pytest.mark.parametrize("k,w_in,w,B", BWD)
def test_lut_backward_bitrows_rows_and_terms(k, w_in, w, B, node):
    Xb = synth.binary_activations(w_in, B, seed=k + 20)
    X8, XW = dev(Xb.astype(np.uint8)), dev(pack_rows(Xb))
    conn = synth.connectivity(w, k, w_in, seed=k + 21)
    theta = synth.table_logits(w, 1 << k, seed=k + 22)
    dY = synth.uniform_gradients(w, B, seed=k + 23, scale=1e-3)
    ref = torch.empty(w, 1 << k, device="cuda")
    bl.bitlogic_lut_backward_u8(X8, dev(conn), dev(theta), ref, node, dY=dev(dY))
    got = torch.full((w, 1 << k), np.nan, device="cuda")
    out = torch.full((w, B), np.nan, device="cuda")
    bl.bitlogic_lut_backward_bitrows(XW, B, dev(conn), dev(theta), got, node, dY=dev(dY), dY_out=out)
    check_exact(got.cpu().numpy(), ref.cpu().numpy(), "dtheta (rows) vs byte rows")
    check_exact(out.cpu().numpy(), dY, "dY_out (rows)")
    wdth, _ = oracle.lut_backward(Xb, conn, theta, dY, want_dx=False, node=node)
    check_grad(got, wdth, "dtheta (rows) vs oracle")
    # a next layer's per-edge terms through its CSR map
    up_w = max(4, w // 2)
    up_conn = synth.connectivity(up_w, 3, w, seed=k + 24)
    off, edge = bl.bitlogic_build_csr(up_conn, w)
    terms = dev(synth.uniform_gradients(up_w * 3, B, seed=k + 25, scale=1e-3))
    ref2 = torch.empty(w, 1 << k, device="cuda")
    out_ref = torch.empty(w, B, device="cuda")
    bl.bitlogic_lut_backward_u8(X8, dev(conn), dev(theta), ref2, node, up_terms=terms, up_off=dev(off),
                                up_edge=dev(edge), dY_out=out_ref)
    got2 = torch.full((w, 1 << k), np.nan, device="cuda")
    out2 = torch.full((w, B), np.nan, device="cuda")
    bl.bitlogic_lut_backward_bitrows(XW, B, dev(conn), dev(theta), got2, node, up_terms=terms, up_off=dev(off),
                                     up_edge=dev(edge), dY_out=out2)
    check_exact(out2.cpu().numpy(), out_ref.cpu().numpy(), "dY_out (terms)")
    check_exact(got2.cpu().numpy(), ref2.cpu().numpy(), "dtheta (terms) vs byte rows")
    assert bl.bitlogic_device_error() == 0


@pytest.mark.parametrize("k", [2, 6])
def test_lut_backward_bitrows_node_order(k):
    # the order in which the warps take the nodes changes no result; an
    # entry outside the nodes is flagged and skipped
    w_in, w, up_w, B = 80, 70, 90, 1028
    Xb = synth.binary_activations(w_in, B, seed=k + 70)
    XW = dev(pack_rows(Xb))
    conn = dev(synth.connectivity(w, k, w_in, seed=k + 71))
    theta = dev(synth.table_logits(w, 1 << k, seed=k + 72))
    up_conn = synth.connectivity(up_w, 4, w, seed=k + 73)
    off, edge = bl.bitlogic_build_csr(up_conn, w)
    terms = dev(synth.uniform_gradients(up_w * 4, B, seed=k + 74, scale=1e-3))
    kw = dict(up_terms=terms, up_off=dev(off), up_edge=dev(edge))
    ref = torch.empty(w, 1 << k, device="cuda")
    out_ref = torch.empty(w, B, device="cuda")
    bl.bitlogic_lut_backward_bitrows(XW, B, conn, theta, ref, dY_out=out_ref, **kw)
    for order in (bl.bitlogic_degree_order(off), np.random.default_rng(k).permutation(w).astype(np.int32)):
        # the next layer's CSR map in the order's sequence: node order[p]'s
        # edges (the same ones, in the same increasing order) at position p
        rank = np.empty_like(order)
        rank[order] = np.arange(w, dtype=np.int32)
        off_o, edge_o = bl.bitlogic_build_csr(rank[up_conn], w)
        np.testing.assert_array_equal(np.diff(off_o), np.diff(off)[order])
        got = torch.full((w, 1 << k), np.nan, device="cuda")
        out = torch.full((w, B), np.nan, device="cuda")
        bl.bitlogic_lut_backward_bitrows(XW, B, conn, theta, got, dY_out=out, order=dev(order), up_terms=terms,
                                         up_off=dev(off_o), up_edge=dev(edge_o))
        check_exact(got.cpu().numpy(), ref.cpu().numpy(), "dtheta (ordered)")
        check_exact(out.cpu().numpy(), out_ref.cpu().numpy(), "dY_out (ordered)")
        # dY rows: the order changes the schedule only
        dY = dev(synth.uniform_gradients(w, B, seed=k + 75, scale=1e-3))
        ref_r = torch.empty(w, 1 << k, device="cuda")
        bl.bitlogic_lut_backward_bitrows(XW, B, conn, theta, ref_r, dY=dY)
        got_r = torch.full((w, 1 << k), np.nan, device="cuda")
        bl.bitlogic_lut_backward_bitrows(XW, B, conn, theta, got_r, dY=dY, order=dev(order))
        check_exact(got_r.cpu().numpy(), ref_r.cpu().numpy(), "dtheta (ordered, dY rows)")
    assert bl.bitlogic_device_error() == 0
    bad = np.arange(w, dtype=np.int32)
    bad[5] = w                                   # one entry past the last node
    got = torch.full((w, 1 << k), np.nan, device="cuda")
    bl.bitlogic_lut_backward_bitrows(XW, B, conn, theta, got, order=dev(bad), **kw)
    assert bl.bitlogic_device_error() == -8
    g = got.cpu().numpy()
    assert np.isnan(g[5]).all()                  # node 5 was never taken
    keep = np.arange(w) != 5
    check_exact(g[keep], ref.cpu().numpy()[keep], "dtheta (other nodes)")


@pytest.mark.parametrize("k,group", [(6, 4), (2, 13)])
def test_lut_backward_bitrows_grouped_rows(k, group):
    w_in, w, B = 90, 52, 2052
    Xb = synth.binary_activations(w_in, B, seed=k + 60)
    conn = synth.connectivity(w, k, w_in, seed=k + 61)
    theta = synth.table_logits(w, 1 << k, seed=k + 62)
    dY = synth.uniform_gradients(w // group, B, seed=k + 63, scale=1e-3)
    ref = torch.empty(w, 1 << k, device="cuda")
    bl.bitlogic_lut_backward_u8(dev(Xb.astype(np.uint8)), dev(conn), dev(theta), ref, dY=dev(dY), dy_group=group)
    got = torch.full((w, 1 << k), np.nan, device="cuda")
    bl.bitlogic_lut_backward_bitrows(dev(pack_rows(Xb)), B, dev(conn), dev(theta), got, dY=dev(dY),
                                     dy_group=group)
    check_exact(got.cpu().numpy(), ref.cpu().numpy(), "dtheta (grouped rows)")
    wdth, _ = oracle.lut_backward(Xb, conn, theta, np.repeat(dY, group, axis=0), want_dx=False)
    check_grad(got, wdth, "dtheta (grouped rows) vs oracle")
    assert bl.bitlogic_device_error() == 0


def test_lut_bitrows_empty_batch_and_ragged_backward():
    k, w_in, w = 3, 20, 6
    conn = dev(synth.connectivity(w, k, w_in, seed=1))
    theta = dev(synth.table_logits(w, 8, seed=2))
    X0 = torch.empty(w_in, 0, dtype=torch.int32, device="cuda")
    bl.bitlogic_lut_forward_bitrows(X0, 0, conn, theta, torch.empty(w, 0, device="cuda"))
    dth = torch.full((w, 8), np.nan, device="cuda")
    bl.bitlogic_lut_backward_bitrows(X0, 0, conn, theta, dth, dY=torch.empty(w, 0, device="cuda"))
    assert torch.all(dth == 0)
    XW = torch.zeros(w_in, bl.bitrow_words(6), dtype=torch.int32, device="cuda")
    with pytest.raises(bl.BitLogicError):   # the backward needs B % 4 == 0
        bl.bitlogic_lut_backward_bitrows(XW, 6, conn, theta, dth, dY=torch.zeros(w, 6, device="cuda"))
