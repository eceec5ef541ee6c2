"""The C ABI without a GPU: the library builds, loads, exports every symbol
``include/bitlogic.h`` declares, and its host-only parts behave."""
import ctypes
import os
import re
import subprocess

import numpy as np
import pytest

import paper_2602_07400_gb300 as bl
from paper_2602_07400_gb300 import synth

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "bitlogic.h")


def _declared():
    src = open(HEADER).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(bitlogic_\w+)\s*\(", src)))


def test_header_declares_the_boundary():
    names = _declared()
    for n in ["bitlogic_encode_thermometer", "bitlogic_lut_forward", "bitlogic_lut_backward",
              "bitlogic_head_loss", "bitlogic_pack_bits", "bitlogic_hard_forward"]:
        assert n in names


def test_library_exports_every_declared_symbol():
    lib = bl.load()
    for n in _declared():
        assert hasattr(lib, n), n
    out = subprocess.run(["nm", "-D", "--defined-only", bl.LIB_PATH], capture_output=True,
                         text=True, check=True).stdout
    exported = set(re.findall(r"\b(bitlogic_\w+)\b", out))
    assert set(_declared()) <= exported


def test_python_binding_names_match_header():
    for n in _declared():
        if n in ("bitlogic_internal_index_error",):
            continue
        assert hasattr(bl, n), n


def test_status_strings_and_version():
    assert bl.bitlogic_status_string(0) == "ok"
    for c in range(-1, -13, -1):
        assert bl.bitlogic_status_string(c) != "unknown status"
    assert bl.bitlogic_version() >= 100


def test_build_csr_matches_inverse_map():
    w, k, w_in = 300, 6, 97
    conn = synth.connectivity(w, k, w_in, seed=5)
    off, edge = bl.bitlogic_build_csr(conn, w_in)
    assert off[0] == 0 and off[-1] == w * k
    flat = conn.reshape(-1)
    for i in range(w_in):
        es = edge[off[i]:off[i + 1]]
        want = np.nonzero(flat == i)[0]
        np.testing.assert_array_equal(es, want)        # increasing edge ids
    # inputs never read get empty rows
    conn2 = np.array([[0, 1], [1, 2]], np.int32)
    off2, edge2 = bl.bitlogic_build_csr(conn2, 6)
    assert off2.tolist() == [0, 1, 3, 4, 4, 4, 4]
    assert edge2.tolist() == [0, 1, 2, 3]


def test_csr_positions_invert_the_edge_map():
    conn = synth.connectivity(200, 6, 97, seed=7)
    off, edge = bl.bitlogic_build_csr(conn, 97)
    pos = bl.bitlogic_csr_positions(edge)
    np.testing.assert_array_equal(pos[edge], np.arange(edge.size))
    np.testing.assert_array_equal(edge[pos], np.arange(edge.size))
    # each input's edges occupy its CSR range
    flat = conn.reshape(-1)
    assert np.all(pos >= off[flat]) and np.all(pos < off[flat + 1])
    for bad in ([0, 0, 1], [0, 3, 1], [-1, 0, 1]):
        with pytest.raises(bl.BitLogicError) as e:
            bl.bitlogic_csr_positions(np.array(bad, np.int32))
        assert e.value.code == -7


def test_build_csr_rejects_out_of_range():
    conn = np.array([[0, 5]], np.int32)
    with pytest.raises(bl.BitLogicError) as e:
        bl.bitlogic_build_csr(conn, 5)
    assert e.value.code == -7
    with pytest.raises(bl.BitLogicError):
        bl.bitlogic_build_csr(np.array([[0, -1]], np.int32), 5)


def test_host_validation_returns_before_any_launch():
    # every call below is rejected on the host, so no CUDA work is issued
    lib = bl.load()
    P = ctypes.c_void_p
    fake = P(16)
    thr = (ctypes.c_uint8 * 3)(64, 128, 192)
    assert lib.bitlogic_lut_forward(None, 4, 8, fake, fake, 2, 2, fake, None) == -1
    assert lib.bitlogic_lut_forward(fake, 4, 8, fake, fake, 2, 7, fake, None) == -3
    assert lib.bitlogic_lut_forward(fake, 4, 8, fake, fake, 2, 0, fake, None) == -3
    assert lib.bitlogic_lut_forward(fake, 2, 8, fake, fake, 2, 3, fake, None) == -3
    assert lib.bitlogic_lut_forward(fake, 0, 8, fake, fake, 2, 2, fake, None) == -2
    assert lib.bitlogic_lut_forward(fake, 4, -1, fake, fake, 2, 2, fake, None) == -2
    # B == 0 is an accepted no-op
    assert lib.bitlogic_lut_forward(fake, 4, 0, fake, fake, 2, 2, fake, None) == 0
    # backward: dX requested without CSR / workspace, too-small / misaligned workspace
    assert lib.bitlogic_lut_backward(fake, 4, 8, fake, fake, 2, 2, fake, None, None,
                                     fake, fake, fake, 1 << 20, None) == -1
    assert lib.bitlogic_lut_backward(fake, 4, 8, fake, fake, 2, 2, fake, fake, fake,
                                     fake, fake, fake, 4, None) == -5
    assert lib.bitlogic_lut_backward(fake, 4, 8, fake, fake, 2, 2, fake, fake, fake,
                                     fake, fake, P(17), 1 << 20, None) == -4
    # issue probe: NULL sink, short sink, negative iterations, unknown kind
    n = lib.bitlogic_issue_probe_threads()
    assert n > 0 and lib.bitlogic_issue_probe_ops_per_iter() > 0
    assert lib.bitlogic_issue_probe_blocks() > 0 and n == 1024 * lib.bitlogic_issue_probe_blocks()
    assert lib.bitlogic_issue_probe(0, 1, 1, None, n, None, None) == -1
    assert lib.bitlogic_issue_probe(0, 1, 1, fake, n - 1, None, None) == -2
    assert lib.bitlogic_issue_probe(0, -1, 1, fake, n, None, None) == -2
    assert lib.bitlogic_issue_probe(0, (1 << 20) + 1, 1, fake, n, None, None) == -2
    assert lib.bitlogic_issue_probe(7, 1, 1, fake, n, None, None) == -2
    # through backward: next-layer fan-in above 3, B not a multiple of 4,
    # group not dividing the next layer, missing inputs
    th = lib.bitlogic_lut_backward_through
    assert th(fake, 8, 8, fake, fake, 8, 2, 0, fake, fake, fake, 8, 4, fake, 1, fake, None, fake, None, None) == -3
    assert th(fake, 8, 6, fake, fake, 8, 2, 0, fake, fake, fake, 8, 2, fake, 1, fake, None, fake, None, None) == -4
    assert th(fake, 8, 8, fake, fake, 8, 2, 0, fake, fake, fake, 8, 2, fake, 3, fake, None, fake, None, None) == -2
    assert th(fake, 8, 8, fake, fake, 8, 2, 0, fake, None, fake, 8, 2, fake, 1, fake, None, fake, None, None) == -1
    assert th(fake, 8, 8, fake, fake, 8, 2, 5, fake, fake, fake, 8, 2, fake, 1, fake, None, fake, None, None) == -12
    # head: w % C != 0, tau <= 0
    assert lib.bitlogic_head_loss(fake, 10, 8, 3, 1.0, fake, None, fake, None, fake, 1 << 20, None) == -2
    assert lib.bitlogic_head_loss(fake, 9, 8, 3, 0.0, fake, None, fake, None, fake, 1 << 20, None) == -2
    # thresholds: b out of range
    assert lib.bitlogic_pack_bits(fake, 64, 4, thr, 0, fake, None) == -9
    assert lib.bitlogic_pack_bits(fake, 64, 4, thr, 33, fake, None) == -9
    assert lib.bitlogic_encode_thermometer(fake, 64, 4, None, 3, fake, None) == -1
    # hard: headless call needs yp; head needs counts and w % C == 0
    assert lib.bitlogic_hard_forward(fake, 8, 64, fake, fake, 4, 2, None, 0, None, None, None) == -1
    assert lib.bitlogic_hard_forward(fake, 8, 64, fake, fake, 4, 2, None, 2, None, None, None) == -1
    assert lib.bitlogic_hard_forward(fake, 8, 64, fake, fake, 4, 2, None, 3, fake, None, None) == -2
    assert lib.bitlogic_binarize_tables(fake, 4, 7, fake, None) == -3
    # AdamW: step >= 1, betas in [0, 1), eps > 0, n >= 0; n == 0 is a no-op
    F = ctypes.c_float
    adamw = lib.bitlogic_adamw_update
    assert adamw(fake, fake, fake, fake, 8, 0, F(0.01), F(0.9), F(0.999), F(1e-8), F(0.0), None) == -11
    assert adamw(fake, fake, fake, fake, 8, 1, F(0.01), F(1.0), F(0.999), F(1e-8), F(0.0), None) == -11
    assert adamw(fake, fake, fake, fake, 8, 1, F(0.01), F(0.9), F(0.999), F(0.0), F(0.0), None) == -11
    assert adamw(fake, fake, fake, fake, -1, 1, F(0.01), F(0.9), F(0.999), F(1e-8), F(0.0), None) == -2
    assert adamw(None, None, None, None, 0, 1, F(0.01), F(0.9), F(0.999), F(1e-8), F(0.0), None) == 0
    assert adamw(None, fake, fake, fake, 8, 1, F(0.01), F(0.9), F(0.999), F(1e-8), F(0.0), None) == -1
    # pixel histogram: negative size, NULL with bytes to count; n == 0 is a no-op
    assert lib.bitlogic_pixel_histogram(fake, -1, fake, None) == -2
    assert lib.bitlogic_pixel_histogram(None, 5, fake, None) == -1
    assert lib.bitlogic_pixel_histogram(fake, 5, None, None) == -1
    assert lib.bitlogic_pixel_histogram(None, 0, None, None) == 0
    # routing: candidates per slot 1..32 and <= w_in, slots > 0, pointers
    rf, rb, rs = lib.bitlogic_route_forward, lib.bitlogic_route_backward, lib.bitlogic_route_snap
    assert rf(fake, 64, 8, fake, fake, 10, 33, fake, None, None) == -3
    assert rf(fake, 64, 8, fake, fake, 10, 0, fake, None, None) == -3
    assert rf(fake, 4, 8, fake, fake, 10, 5, fake, None, None) == -3
    assert rf(fake, 64, 8, fake, fake, 0, 4, fake, None, None) == -2
    assert rf(fake, 64, 8, None, fake, 10, 4, fake, None, None) == -1
    assert rf(fake, 64, 8, fake, fake, 10, 4, None, None, None) == -1
    assert rf(fake, 64, 0, fake, fake, 10, 4, None, None, None) == 0
    assert rb(fake, 64, 8, fake, fake, 10, 4, fake, None, None, None, None, None, None) == -1
    assert rb(fake, 64, 8, fake, fake, 10, 4, fake, fake, None, fake, fake, fake, None) == -1
    assert rs(fake, fake, 10, 0, fake, None) == -3
    assert rs(fake, fake, 0, 4, fake, None) == -2
    assert rs(None, fake, 10, 4, fake, None) == -1
    assert lib.bitlogic_route_forward_u8(fake, 64, 8, fake, fake, 10, 33, fake, None, None) == -3
    assert lib.bitlogic_route_backward_u8(fake, 64, 8, fake, fake, 10, 4, fake, None, None) == -1
    assert lib.bitlogic_encode_thermometer_u8(fake, 64, 4, thr, 0, fake, None) == -9
    # node form: only soft (0) and straight-through (1)
    fwd_node, bwd_node = lib.bitlogic_lut_forward_node, lib.bitlogic_lut_backward_node
    assert fwd_node(fake, 8, 64, fake, fake, 4, 2, 2, fake, None) == -12
    assert fwd_node(fake, 8, 64, fake, fake, 4, 2, -1, fake, None) == -12
    assert fwd_node(fake, 8, 64, fake, fake, 4, 7, 1, fake, None) == -3
    assert bwd_node(fake, 8, 64, fake, fake, 4, 2, 2, fake, 1, None, None, None, 0, fake, None, None,
                    None, None) == -12
    with pytest.raises(ValueError):
        bl.bitlogic_lut_forward_node(None, None, None, None, node="hard")
    # forward on byte rows: node form, fan-in, shapes, NULLs (B = 0 is a no-op)
    fwd_u8 = lib.bitlogic_lut_forward_u8
    assert fwd_u8(fake, 8, 64, fake, fake, 4, 2, 2, fake, None) == -12
    assert fwd_u8(fake, 8, 64, fake, fake, 4, 7, 0, fake, None) == -3
    assert fwd_u8(fake, 8, 64, fake, fake, 4, 9, 0, fake, None) == -3   # k > w_in
    assert fwd_u8(fake, 0, 64, fake, fake, 4, 2, 0, fake, None) == -2
    assert fwd_u8(fake, 8, -1, fake, fake, 4, 2, 0, fake, None) == -2
    assert fwd_u8(None, 8, 64, fake, fake, 4, 2, 0, fake, None) == -1
    assert fwd_u8(fake, 8, 64, fake, fake, 4, 2, 0, None, None) == -1
    assert fwd_u8(fake, 8, 64, None, fake, 4, 2, 0, fake, None) == -1
    assert fwd_u8(None, 8, 0, fake, fake, 4, 2, 0, None, None) == 0
    # wire bit rows: encoder thresholds and shapes, forward and backward
    # checks as on byte rows, 4-byte aligned words, B % 4 == 0 for the
    # backward (B = 0 is a no-op)
    enc_b, fwd_b, bwd_b = (lib.bitlogic_encode_thermometer_bitrows, lib.bitlogic_lut_forward_bitrows,
                           lib.bitlogic_lut_backward_bitrows)
    assert enc_b(fake, 64, 4, thr, 0, fake, None) == -9
    assert enc_b(fake, 64, 0, thr, 3, fake, None) == -2
    assert enc_b(None, 64, 4, thr, 3, fake, None) == -1
    assert enc_b(None, 0, 4, thr, 3, None, None) == 0
    assert fwd_b(fake, 8, 64, fake, fake, 4, 2, 2, fake, None) == -12
    assert fwd_b(fake, 8, 64, fake, fake, 4, 7, 0, fake, None) == -3
    assert fwd_b(fake, 0, 64, fake, fake, 4, 2, 0, fake, None) == -2
    assert fwd_b(None, 8, 64, fake, fake, 4, 2, 0, fake, None) == -1
    assert fwd_b(P(18), 8, 64, fake, fake, 4, 2, 0, fake, None) == -4
    assert fwd_b(None, 8, 0, fake, fake, 4, 2, 0, None, None) == 0
    assert bwd_b(fake, 8, 64, fake, fake, 4, 2, 0, None, 1, None, None, None, 0, None, fake, None, None) == -1
    assert bwd_b(fake, 8, 64, fake, fake, 4, 2, 0, fake, 1, fake, fake, None, 4, None, fake, None, None) == -1
    assert bwd_b(fake, 8, 64, fake, fake, 4, 2, 0, fake, 3, None, None, None, 0, None, fake, None, None) == -2
    assert bwd_b(fake, 8, 66, fake, fake, 4, 2, 0, fake, 1, None, None, None, 0, None, fake, None, None) == -4
    assert bwd_b(fake, 8, 64, fake, fake, 4, 2, 2, fake, 1, None, None, None, 0, None, fake, None, None) == -12


@pytest.mark.parametrize("n,b,seed", [(1, 1, 0), (5, 4, 1), (1000, 8, 2), (65537, 32, 3), (300, 15, 4)])
def test_quantile_thresholds_from_a_histogram_match_the_oracle(n, b, seed):
    # host-only step of the quantile fit: thresholds from 256 counts
    import oracle
    rng = np.random.default_rng(seed)
    x = rng.integers(0, 256, size=n, dtype=np.uint8)
    if seed % 2:
        x[rng.random(n) < 0.8] = 0               # a point mass, as in digit images
    hist = np.bincount(x, minlength=256).astype(np.uint64)
    np.testing.assert_array_equal(bl.bitlogic_quantile_thresholds(hist, b), oracle.quantile_thresholds(x, b))


def test_degree_order_is_a_stable_sort_by_decreasing_degree():
    # host helper: nodes by decreasing CSR degree, ties in increasing index
    rng = np.random.default_rng(3)
    for w, w_in, k in ((50, 40, 3), (300, 1000, 6), (7, 7, 1)):
        conn = rng.integers(0, w_in, size=(w, k)).astype(np.int32)
        off, _ = bl.bitlogic_build_csr(conn, w_in)
        deg = np.diff(off)
        order = bl.bitlogic_degree_order(off)
        np.testing.assert_array_equal(order, np.argsort(-deg, kind="stable"))
        assert sorted(order.tolist()) == list(range(w_in))
    lib = bl.load()
    P = ctypes.c_void_p
    off = np.array([0, 2, 1], np.int32)               # decreasing: not a CSR map
    out = np.zeros(2, np.int32)
    assert lib.bitlogic_degree_order(off.ctypes.data_as(P), 2, out.ctypes.data_as(P)) == -7
    off = np.array([1, 2, 3], np.int32)               # does not start at 0
    assert lib.bitlogic_degree_order(off.ctypes.data_as(P), 2, out.ctypes.data_as(P)) == -7
    assert lib.bitlogic_degree_order(off.ctypes.data_as(P), 0, out.ctypes.data_as(P)) == -2
    assert lib.bitlogic_degree_order(None, 2, out.ctypes.data_as(P)) == -1


def test_quantile_thresholds_rejects_bad_input():
    with pytest.raises(bl.BitLogicError):
        bl.bitlogic_quantile_thresholds(np.zeros(256, np.uint64), 4)    # empty
    with pytest.raises(bl.BitLogicError):
        bl.bitlogic_quantile_thresholds(np.ones(256, np.uint64), 33)    # b > 32
    with pytest.raises(bl.BitLogicError):
        bl.bitlogic_quantile_thresholds(np.ones(256, np.uint64), 0)


def test_workspace_queries():
    assert bl.bitlogic_lut_backward_workspace(100, 64, 10, 6, False) == 0
    assert bl.bitlogic_lut_backward_workspace(100, 64, 10, 6, True) == 10 * 6 * 64 * 4
    assert bl.bitlogic_head_loss_workspace(64, 10) >= 2 * 64 * 10 * 4 + 64 * 4


def test_no_cpu_fallback_without_the_library(monkeypatch):
    # with the shared library absent (and building switched off) the binding
    # raises instead of computing anything another way
    missing = os.path.join(ROOT, "no_such_dir", "libbitlogic.so")
    monkeypatch.setattr(bl, "_lib", None)
    monkeypatch.setattr(bl, "LIB_PATH", missing)
    monkeypatch.setattr(bl._build, "LIB", missing)
    with pytest.raises(RuntimeError):
        bl.load(build_if_missing=False)


def test_compute_calls_reject_host_tensors():
    # every compute call takes device tensors only: host tensors are refused
    # before any launch, so there is no CPU path to fall back on
    import torch
    x = torch.zeros(4, 8, dtype=torch.uint8)
    X = torch.zeros(16, 4)
    conn = torch.zeros(2, 2, dtype=torch.int32)
    theta = torch.zeros(2, 4)
    with pytest.raises(ValueError, match="CUDA"):
        bl.bitlogic_encode_thermometer(x, [64, 128], torch.zeros(16, 4))
    with pytest.raises(ValueError, match="CUDA"):
        bl.bitlogic_lut_forward(X, conn, theta, torch.zeros(2, 4))
    with pytest.raises(ValueError, match="CUDA"):
        bl.bitlogic_pack_bits(x, [64, 128], torch.zeros(16, 1, dtype=torch.int32))
    with pytest.raises(ValueError, match="CUDA"):
        bl.bitlogic_issue_probe("lop3", 1, torch.zeros(8, dtype=torch.int32))
