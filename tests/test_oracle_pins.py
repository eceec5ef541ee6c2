"""Pins of the CPU oracle to what the paper and the mathematics fix.

Each test checks the oracle against something other than itself: a
hand-worked value under ``tests/golden/``, a closed form, an invariant, a
library routine (torch autograd / cross-entropy), finite differences, or an
independent brute force.  Every plausible slip (a swapped slot/bit order, a
dropped term, a wrong sign, a transposed layout) fails at least one of them.
"""
import math
import os

import numpy as np
import pytest
import torch

import oracle
from paper_2602_07400_gb300 import synth

GOLD = os.path.join(os.path.dirname(__file__), "golden")


def _gold_lines(name):
    with open(os.path.join(GOLD, name)) as f:
        return [ln.split() for ln in f if ln.strip() and not ln.startswith("#")]


def _sig(z):
    return 1.0 / (1.0 + np.exp(-np.asarray(z, np.float64)))


# ---------------------------------------------------------------- encoder --

def test_linear_thresholds_reading():
    # b equispaced thresholds at i/(b+1) of the uint8 range (App. A); the
    # workloads' literal threshold sets must be this reading
    assert oracle.linear_thresholds(3).tolist() == [64, 128, 192]
    assert oracle.linear_thresholds(7).tolist() == [32 * i for i in range(1, 8)]
    assert oracle.linear_thresholds(15).tolist() == [16 * i for i in range(1, 16)]
    for wl in synth.WORKLOADS.values():
        assert list(wl.thresholds) == oracle.linear_thresholds(wl.b).tolist()


def test_encoder_golden():
    rows = _gold_lines("thermometer_b3.txt")
    px = np.array([int(r[0]) for r in rows], np.uint8)
    want = np.array([[int(v) for v in r[1:]] for r in rows], np.float64)
    bits = oracle.encode_thermometer(px.reshape(-1, 1), [64, 128, 192])
    assert bits.shape == (3, px.size)
    np.testing.assert_array_equal(bits.T, want)


def test_encoder_unary_code_and_layout():
    rng = np.random.default_rng(1)
    x = rng.integers(0, 256, size=(37, 5), dtype=np.uint8)
    thr = [32 * i for i in range(1, 8)]
    bits = oracle.encode_thermometer(x, thr).reshape(5, 7, 37)  # [j][i][s]
    ones = bits.sum(axis=1)                                     # [j][s]
    # ones-count = #{i : T_i < v}
    want = (x.T[:, None, :] > np.array(thr)[None, :, None]).sum(axis=1)
    np.testing.assert_array_equal(ones, want)
    # unary (thermometer) code: wire i+1 set implies wire i set
    assert np.all(bits[:, :-1, :] >= bits[:, 1:, :])
    # feature-major wire order j*b + i
    j, i, s = 3, 4, 11
    assert bits[j, i, s] == float(x[s, j] > thr[i])


# ------------------------------------------------ quantile thermometer fit --
#
# Distributive thermometer (§3, App. A, App. B): thresholds at the empirical
# quantiles i/(b+1) of the flattened training pixels.

def _np_quantile_thresholds(x, b):
    # numpy's linear-interpolation quantile on the pixel scale, then the
    # floor that the strict integer compare implies; the true fractional
    # part is 0 or at least 1/(b+1), so a 1e-9 nudge only absorbs rounding
    q = np.quantile(np.asarray(x, np.float64).reshape(-1), [i / (b + 1) for i in range(1, b + 1)],
                    method="linear")
    return np.floor(q + 1e-9).astype(np.int64), q


@pytest.mark.parametrize("n,b,seed", [(1, 3, 0), (2, 4, 1), (3, 7, 2), (7, 15, 3), (1000, 4, 4),
                                      (4097, 8, 5), (100003, 32, 6), (256, 1, 7)])
def test_quantile_fit_matches_numpy(n, b, seed):
    rng = np.random.default_rng(seed)
    x = rng.integers(0, 256, size=n, dtype=np.uint8)
    got = oracle.quantile_thresholds(x, b)
    want, q = _np_quantile_thresholds(x, b)
    np.testing.assert_array_equal(got.astype(np.int64), want)
    # the stored integer threshold encodes exactly as the real quantile
    v = np.arange(256)[:, None]
    np.testing.assert_array_equal(v > got[None, :].astype(np.int64), v > q[None, :] + 1e-9)


def test_quantile_fit_collapses_on_a_point_mass_at_zero():
    # the MNIST observation of App. B: with a point mass at zero between the
    # 7/9 and 8/9 quantiles, b = 4 gives four zero thresholds (every wire is
    # pixel > 0) and b = 8 seven zeros and a last threshold above zero
    rng = np.random.default_rng(11)
    n = 200000
    x = np.where(rng.random(n) < 0.83, 0, rng.integers(1, 256, size=n)).astype(np.uint8)
    assert list(oracle.quantile_thresholds(x, 4)) == [0, 0, 0, 0]
    t8 = oracle.quantile_thresholds(x, 8)
    assert list(t8[:7]) == [0] * 7 and t8[7] > 0
    # the collapsed encoder emits b identical wires per feature
    bits = oracle.encode_thermometer(x[:64].reshape(8, 8), oracle.quantile_thresholds(x, 4))
    w = bits.reshape(8, 4, 8)
    assert np.all(w == w[:, :1, :])


def test_quantile_fit_on_a_flat_histogram_is_near_linear():
    # every value equally often: the quantile at level p is 255 p up to the
    # one-step interpolation between neighbouring values
    x = np.repeat(np.arange(256, dtype=np.uint8), 50)
    for b in (3, 7, 15):
        t = oracle.quantile_thresholds(x, b).astype(np.float64)
        assert np.all(np.abs(t - 255.0 * np.arange(1, b + 1) / (b + 1)) <= 1.0)
    # a constant image: every threshold is that constant
    assert list(oracle.quantile_thresholds(np.full(99, 37, np.uint8), 5)) == [37] * 5


# ----------------------------------------------------------- soft forward --

def test_soft_node_golden_k2():
    g = {r[0]: [float(v) for v in r[1:]] for r in _gold_lines("lightlut_k2_worked.txt")}
    theta = np.array(g["theta"], np.float32).reshape(1, 4)
    X = np.array(g["x"], np.float64).reshape(2, 1)
    conn = np.array([[0, 1]], np.int32)
    Y = oracle.lut_forward(X, conn, theta)
    # theta is stored in fp32, so t differs from the exact fractions at 1e-8
    assert Y[0, 0] == pytest.approx(g["y"][0], abs=1e-7)
    dth, dX = oracle.lut_backward(X, conn, theta, np.ones((1, 1)))
    np.testing.assert_allclose(dX[:, 0], g["dx"], atol=1e-7)
    np.testing.assert_allclose(dth[0], g["dtheta"], atol=1e-7)
    # binary inputs pick one table entry: (1,0) -> t1, (0,1) -> t2
    Xb = np.array([[1.0, 0.0], [0.0, 1.0]])
    Yb = oracle.lut_forward(Xb, conn, theta)
    np.testing.assert_allclose(Yb[0], _sig(theta[0, [1, 2]]), rtol=1e-14)


@pytest.mark.parametrize("k", [1, 2, 3, 4, 6])
def test_binary_inputs_return_table_entry(k):
    # on {0,1} inputs a soft node returns exactly its table entry (every
    # surrogate discretizes to the same truth table, §3); slot i = bit i
    rng = np.random.default_rng(k)
    w_in, w, B = 13, 7, 29
    X = rng.integers(0, 2, size=(w_in, B)).astype(np.float64)
    conn = synth.connectivity(w, k, w_in, seed=k)
    theta = synth.table_logits(w, 1 << k, seed=10 + k)
    Y = oracle.lut_forward(X, conn, theta)
    idx = np.zeros((w, B), np.int64)
    for i in range(k):
        idx |= X[conn[:, i], :].astype(np.int64) << i
    want = _sig(np.take_along_axis(theta, idx, axis=1))
    np.testing.assert_allclose(Y, want, rtol=1e-14, atol=0)


def test_k1_is_a_lerp():
    theta = np.array([[0.3, -1.7]], np.float32)
    t = _sig(theta[0])
    X = np.linspace(0, 1, 11).reshape(1, -1)
    Y = oracle.lut_forward(X, np.array([[0]], np.int32), theta)
    np.testing.assert_allclose(Y[0], (1 - X[0]) * t[0] + X[0] * t[1], rtol=1e-14)


def test_k2_closed_form():
    rng = np.random.default_rng(5)
    theta = rng.standard_normal((1, 4)).astype(np.float32)
    t = _sig(theta[0])
    X = rng.random((2, 50))
    Y = oracle.lut_forward(X, np.array([[0, 1]], np.int32), theta)[0]
    x0, x1 = X
    want = (t[0] * (1 - x0) * (1 - x1) + t[1] * x0 * (1 - x1)
            + t[2] * (1 - x0) * x1 + t[3] * x0 * x1)
    np.testing.assert_allclose(Y, want, rtol=1e-13)


@pytest.mark.parametrize("k", [2, 4, 6])
def test_multilinear_in_each_input(k):
    rng = np.random.default_rng(20 + k)
    theta = synth.table_logits(3, 1 << k, seed=k)
    conn = np.array([rng.permutation(k) for _ in range(3)], np.int32)
    base = rng.random((k, 1))
    for i in range(k):
        a = rng.random()
        cols = np.repeat(base, 3, axis=1)
        cols[i, 0], cols[i, 1], cols[i, 2] = 0.0, 1.0, a
        Y = oracle.lut_forward(cols, conn, theta)
        np.testing.assert_allclose(Y[:, 2], (1 - a) * Y[:, 0] + a * Y[:, 1], rtol=1e-12)


def test_partition_of_unity():
    # constant table -> constant output, zero input gradient
    k, w, B = 6, 4, 17
    rng = np.random.default_rng(3)
    X = rng.random((9, B))
    conn = synth.connectivity(w, k, 9, seed=3)
    c = np.array([0.7, -2.0, 0.0, 5.0], np.float32)
    theta = np.repeat(c[:, None], 1 << k, axis=1)
    Y = oracle.lut_forward(X, conn, theta)
    np.testing.assert_allclose(Y, np.repeat(_sig(c)[:, None], B, axis=1), rtol=1e-13)
    _, dX = oracle.lut_backward(X, conn, theta, rng.standard_normal((w, B)))
    np.testing.assert_allclose(dX, 0.0, atol=1e-13)


# ---------------------------------------------------------------- backward --

@pytest.mark.parametrize("k", [1, 2, 3, 4, 6])
def test_finite_differences(k):
    rng = np.random.default_rng(100 + k)
    w_in, w, B = max(k + 2, 8), 5, 4
    X = rng.random((w_in, B))
    conn = synth.connectivity(w, k, w_in, seed=k + 7)
    theta = synth.table_logits(w, 1 << k, seed=k + 8)
    R = rng.standard_normal((w, B))

    def L(Xv, th):
        return float(np.sum(R * oracle.lut_forward(Xv, conn, th)))

    dth, dX = oracle.lut_backward(X, conn, theta, R)
    # dX: the loss is linear in each single input value, so central
    # differences are exact up to rounding
    h = 1e-3
    for (p, s) in [(0, 0), (conn[0, -1], 3), (w_in - 1, 1), (conn[w - 1, 0], 2)]:
        Xp, Xm = X.copy(), X.copy()
        Xp[p, s] += h
        Xm[p, s] -= h
        fd = (L(Xp, theta) - L(Xm, theta)) / (2 * h)
        assert dX[p, s] == pytest.approx(fd, rel=1e-9, abs=1e-12)
    # dtheta: theta is fp32, so use the exact perturbation that fp32 stores
    for (j, a) in [(0, 0), (1, (1 << k) - 1), (w - 1, (1 << k) // 2), (2, 1 % (1 << k))]:
        tp, tm = theta.copy(), theta.copy()
        tp[j, a] = np.float32(theta[j, a] + np.float32(1e-2))
        tm[j, a] = np.float32(theta[j, a] - np.float32(1e-2))
        hp = float(tp[j, a]) - float(theta[j, a])
        hm = float(theta[j, a]) - float(tm[j, a])
        fd = (L(X, tp) - L(X, tm)) / (hp + hm)
        assert dth[j, a] == pytest.approx(fd, rel=2e-5, abs=1e-9)


def test_dtheta_identity():
    # sum_a dtheta[a] / (t_a (1 - t_a)) = sum_s dY[s]   (sum_a w_a = 1)
    rng = np.random.default_rng(9)
    X = rng.random((20, 33))
    conn = synth.connectivity(6, 6, 20, seed=9)
    theta = synth.table_logits(6, 64, seed=9)
    dY = rng.standard_normal((6, 33))
    dth, _ = oracle.lut_backward(X, conn, theta, dY, want_dx=False)
    t = _sig(theta)
    np.testing.assert_allclose((dth / (t * (1 - t))).sum(axis=1), dY.sum(axis=1), rtol=1e-10)


def test_dx_scatter_is_sum_over_consumers():
    # an input read by no node gets zero gradient; one read by two nodes gets
    # the sum of what each node alone would send it
    k, B = 2, 6
    rng = np.random.default_rng(4)
    X = rng.random((5, B))
    conn = np.array([[0, 1], [1, 2]], np.int32)   # input 1 shared, 3 and 4 unused
    theta = synth.table_logits(2, 4, seed=4)
    dY = rng.standard_normal((2, B))
    _, dX = oracle.lut_backward(X, conn, theta, dY)
    _, dA = oracle.lut_backward(X, conn[:1], theta[:1], dY[:1])
    _, dB = oracle.lut_backward(X, conn[1:], theta[1:], dY[1:])
    np.testing.assert_allclose(dX, dA + dB, rtol=1e-13, atol=1e-15)
    assert np.all(dX[3:] == 0.0)


# ------------------------------------------ straight-through hard node --
#
# LightLUT's hard form (§2 "Gradient-based LUT methods", §4 "Node
# parameterization"): the forward samples each table entry as [theta > 0];
# the straight-through estimator sends the table gradient to theta through
# the sigmoid.

def _shannon_forward_torch(X, conn, t):
    """y_j = the node's table folded one input at a time (slot i = bit i of
    the entry index): a different formulation from the oracle's sum of
    corner weights."""
    w, k = conn.shape
    xs = X[torch.as_tensor(conn, dtype=torch.long)]      # [w, k, B]
    B = X.shape[1]
    T = t.reshape((w,) + (2,) * k).unsqueeze(1).expand((w, B) + (2,) * k)
    for i in range(k):   # the last axis is the lowest remaining index bit
        xi = xs[:, i, :].reshape((w, B) + (1,) * (k - 1 - i))
        T = T[..., 0] * (1 - xi) + T[..., 1] * xi
    return T


@pytest.mark.parametrize("k", [1, 2, 4, 6])
def test_st_backward_matches_torch_straight_through(k):
    # torch autograd through t = sigmoid(theta) + ([theta > 0] - sigmoid(theta)).detach()
    rng = np.random.default_rng(500 + k)
    w_in, w, B = max(k + 3, 9), 7, 5
    X = rng.random((w_in, B))
    conn = synth.connectivity(w, k, w_in, seed=k + 50)
    theta = synth.table_logits(w, 1 << k, seed=k + 51)
    theta[0, 0] = 0.0                        # a tie samples 0
    dY = rng.standard_normal((w, B))
    Xt = torch.tensor(X, dtype=torch.float64, requires_grad=True)
    tht = torch.tensor(theta.astype(np.float64), requires_grad=True)
    sg = torch.sigmoid(tht)
    t = sg + ((tht > 0).to(torch.float64) - sg).detach()
    Y = _shannon_forward_torch(Xt, conn, t)
    (Y * torch.tensor(dY)).sum().backward()
    np.testing.assert_allclose(oracle.lut_forward(X, conn, theta, "st"), Y.detach().numpy(),
                               rtol=1e-13, atol=1e-15)
    dth, dX = oracle.lut_backward(X, conn, theta, dY, node="st")
    np.testing.assert_allclose(dth, tht.grad.numpy(), rtol=1e-12, atol=1e-15)
    np.testing.assert_allclose(dX, Xt.grad.numpy(), rtol=1e-12, atol=1e-14)


@pytest.mark.parametrize("k", [2, 4, 6])
def test_st_forward_is_the_saturated_soft_forward(k):
    # tables at theta = +-800 have sigmoid exactly 1 / 0 in double, so the
    # soft forward on them is the hard-sampled forward, on any inputs
    rng = np.random.default_rng(600 + k)
    w_in, w, B = 40, 17, 9
    X = rng.random((w_in, B))
    conn = synth.connectivity(w, k, w_in, seed=k + 60)
    theta = synth.table_logits(w, 1 << k, seed=k + 61)
    sat = np.where(theta > 0, 800.0, -800.0).astype(np.float32)
    np.testing.assert_array_equal(oracle.lut_forward(X, conn, theta, "st"),
                                  oracle.lut_forward(X, conn, sat, "soft"))
    # the input gradient is the soft one of the saturated tables; dtheta keeps
    # the sigmoid slope of the real logits
    dY = rng.standard_normal((w, B))
    dth, dX = oracle.lut_backward(X, conn, theta, dY, node="st")
    _, dXs = oracle.lut_backward(X, conn, sat, dY, node="soft")
    np.testing.assert_allclose(dX, dXs, rtol=1e-13, atol=1e-15)
    dths, _ = oracle.lut_backward(X, conn, theta, dY, want_dx=False, node="soft")
    np.testing.assert_array_equal(dth, dths)


@pytest.mark.parametrize("k", [2, 4, 6])
def test_st_binary_inputs_give_the_hard_lookup(k):
    # on binary inputs the straight-through forward is the deployed network:
    # the bit-packed lookup of the discretized tables (App. C.1)
    rng = np.random.default_rng(700 + k)
    w_in, w, N = 45, 29, 70
    Xb = rng.integers(0, 2, size=(w_in, N)).astype(np.float64)
    conn = synth.connectivity(w, k, w_in, seed=k + 70)
    theta = synth.table_logits(w, 1 << k, seed=k + 71)
    y = oracle.lut_forward(Xb, conn, theta, "st")
    W = (N + 31) // 32
    xp = np.zeros((w_in, W), np.uint32)
    for s in range(N):
        xp[:, s // 32] |= (Xb[:, s].astype(np.uint32) << np.uint32(s % 32))
    yp = oracle.hard_forward(xp, N, conn, oracle.binarize_tables(theta))
    np.testing.assert_array_equal(_unpack(yp, N), y)


def test_st_k1_closed_form():
    # k = 1, theta = (0, 2): y = [0 > 0] (1 - x) + [2 > 0] x = x;
    # dtheta = (s'(0) sum g (1 - x), s'(2) sum g x), s' = s (1 - s); dx = g (1 - 0)
    X = np.array([[0.25, 0.5, 1.0]])
    conn = np.array([[0]], np.int32)
    theta = np.array([[0.0, 2.0]], np.float32)
    g = np.array([[1.0, -2.0, 0.5]])
    np.testing.assert_array_equal(oracle.lut_forward(X, conn, theta, "st"), X)
    dth, dX = oracle.lut_backward(X, conn, theta, g, node="st")
    s2 = 1.0 / (1.0 + math.exp(-2.0))
    want = [0.25 * float(np.sum(g * (1 - X))), s2 * (1 - s2) * float(np.sum(g * X))]
    np.testing.assert_allclose(dth[0], want, rtol=1e-14)
    np.testing.assert_allclose(dX, g, rtol=1e-14)


# ------------------------------------------------------ learnable routing --
#
# Per-slot candidate pools with softmax routing logits (§3 "Connectivity",
# App. A "Initialization"); the slot input is the expected selection.

def test_route_zero_logits_average_the_pool():
    # logits initialised to zero: the uniform expected selection
    rng = np.random.default_rng(1)
    X = rng.random((30, 7))
    cand = synth.candidate_pools(12, 8, 30, seed=2)
    Xr, p = oracle.route_forward(X, cand, np.zeros((12, 8), np.float32))
    np.testing.assert_allclose(p, 1.0 / 8, rtol=1e-15)
    np.testing.assert_allclose(Xr, X[cand].mean(axis=1), rtol=1e-14)


def test_route_saturated_logits_select_one_candidate():
    rng = np.random.default_rng(3)
    X = rng.random((40, 9))
    cand = synth.candidate_pools(10, 16, 40, seed=4)
    r = np.zeros((10, 16), np.float32)
    pick = rng.integers(0, 16, size=10)
    r[np.arange(10), pick] = 60.0
    Xr, _ = oracle.route_forward(X, cand, r)
    np.testing.assert_allclose(Xr, X[cand[np.arange(10), pick]], rtol=0, atol=1e-24)
    np.testing.assert_array_equal(oracle.route_snap(cand, r), cand[np.arange(10), pick])


def test_route_snap_takes_the_first_maximum():
    cand = np.array([[5, 6, 7, 8], [1, 2, 3, 4]], np.int32)
    r = np.array([[0.5, 2.0, 2.0, -1.0], [-3.0, -3.0, -3.0, -3.0]], np.float32)
    np.testing.assert_array_equal(oracle.route_snap(cand, r), [6, 1])


@pytest.mark.parametrize("k,Kc", [(2, 4), (4, 16), (6, 8)])
def test_routed_layer_matches_torch_autograd(k, Kc):
    # routing then a soft node over the slot inputs, against torch autograd
    # through torch.softmax, an index gather and the Shannon-expansion node
    rng = np.random.default_rng(800 + k)
    w_in, w, B = 50, 6, 5
    X = rng.random((w_in, B))
    cand = synth.candidate_pools(w * k, Kc, w_in, seed=k)
    r = synth.table_logits(w * k, Kc, seed=k + 1)
    theta = synth.table_logits(w, 1 << k, seed=k + 2)
    dY = rng.standard_normal((w, B))
    ident = np.arange(w * k, dtype=np.int32).reshape(w, k)
    Xr, _ = oracle.route_forward(X, cand, r)
    dth, G = oracle.lut_backward(Xr, ident, theta, dY)
    dr, dX = oracle.route_backward(X, cand, r, G)
    Xt = torch.tensor(X, requires_grad=True)
    rt = torch.tensor(r.astype(np.float64), requires_grad=True)
    tht = torch.tensor(theta.astype(np.float64), requires_grad=True)
    P = torch.softmax(rt, dim=1)
    Xrt = (P[:, :, None] * Xt[torch.as_tensor(cand, dtype=torch.long)]).sum(dim=1)
    Y = _shannon_forward_torch(Xrt, ident, torch.sigmoid(tht))
    (Y * torch.tensor(dY)).sum().backward()
    np.testing.assert_allclose(Xr, Xrt.detach().numpy(), rtol=1e-13, atol=1e-15)
    np.testing.assert_allclose(dth, tht.grad.numpy(), rtol=1e-11, atol=1e-15)
    np.testing.assert_allclose(dr, rt.grad.numpy(), rtol=1e-10, atol=1e-14)
    np.testing.assert_allclose(dX, Xt.grad.numpy(), rtol=1e-11, atol=1e-14)


def test_route_finite_differences_and_gradient_mass():
    rng = np.random.default_rng(21)
    w_in, n, Kc, B = 20, 9, 6, 4
    X = rng.random((w_in, B))
    cand = synth.candidate_pools(n, Kc, w_in, seed=5)
    r = synth.table_logits(n, Kc, seed=6)
    G = rng.standard_normal((n, B))

    def L(Xv, rv):
        return float(np.sum(G * oracle.route_forward(Xv, cand, rv)[0]))

    dr, dX = oracle.route_backward(X, cand, r, G)
    for (e, m) in [(0, 0), (4, 5), (n - 1, 2)]:
        rp, rm = r.copy(), r.copy()
        rp[e, m] = np.float32(r[e, m] + np.float32(1e-2))
        rm[e, m] = np.float32(r[e, m] - np.float32(1e-2))
        fd = (L(X, rp) - L(X, rm)) / (float(rp[e, m]) - float(rm[e, m]))
        assert dr[e, m] == pytest.approx(fd, rel=2e-5, abs=1e-9)
    h = 1e-3
    for (c, s) in [(cand[0, 0], 0), (cand[3, 2], 3), (w_in - 1, 1)]:
        Xp, Xm = X.copy(), X.copy()
        Xp[c, s] += h
        Xm[c, s] -= h
        assert dX[c, s] == pytest.approx((L(Xp, r) - L(Xm, r)) / (2 * h), rel=1e-9, abs=1e-12)
    # the probabilities of a slot sum to one: the input gradient carries the
    # slot gradients' total, and the logit gradients of a slot sum to zero
    np.testing.assert_allclose(dX.sum(axis=0), G.sum(axis=0), rtol=1e-12)
    np.testing.assert_allclose(dr.sum(axis=1), 0.0, atol=1e-13)


# -------------------------------------------------------------------- head --

def test_head_matches_torch_autograd():
    # group sums / tau -> cross-entropy (mean) against torch's own routine
    rng = np.random.default_rng(11)
    C, g, B, tau = 4, 5, 9, 3.0
    Y = rng.random((C * g, B))
    labels = rng.integers(0, C, size=B).astype(np.int32)
    logits, loss, dY = oracle.head_loss(Y, labels, C, tau)
    Yt = torch.tensor(Y, dtype=torch.float64, requires_grad=True)
    lt = Yt.view(C, g, B).sum(dim=1).t() / tau
    lo = torch.nn.functional.cross_entropy(lt, torch.tensor(labels, dtype=torch.int64))
    lo.backward()
    np.testing.assert_allclose(logits, lt.detach().numpy(), rtol=1e-13)
    assert loss == pytest.approx(lo.item(), rel=1e-13)
    np.testing.assert_allclose(dY, Yt.grad.numpy(), rtol=1e-11, atol=1e-16)


def test_head_closed_forms():
    C, g, B = 10, 3, 7
    # equal group sums -> every logit equal -> loss = ln C
    Y = np.full((C * g, B), 0.25)
    labels = np.arange(B, dtype=np.int32) % C
    _, loss, dY = oracle.head_loss(Y, labels, C, 2.0)
    assert loss == pytest.approx(math.log(C), rel=1e-14)
    # sum over classes of dlogit is zero; dlogit[label] = (1/C - 1)/B
    dl = dY.reshape(C, g, B)[:, 0, :] * 2.0
    np.testing.assert_allclose(dl.sum(axis=0), 0.0, atol=1e-15)
    assert dl[labels[0], 0] == pytest.approx((1.0 / C - 1.0) / B, rel=1e-12)
    # one dominant logit on the label -> loss -> 0
    Y2 = np.zeros((C * g, B))
    for s in range(B):
        Y2[labels[s] * g:(labels[s] + 1) * g, s] = 1.0
    _, loss2, _ = oracle.head_loss(Y2, labels, C, 0.05)
    assert loss2 < 1e-20


def test_full_step_finite_differences():
    # the whole chain (encoder -> 2 layers -> head + CE -> backward) against
    # central differences of the loss in a few layer-1 and layer-2 logits
    rng = np.random.default_rng(12)
    B, d, C = 6, 5, 2
    x = rng.integers(0, 256, size=(B, d), dtype=np.uint8)
    labels = rng.integers(0, C, size=B).astype(np.int32)
    thr = [64, 128, 192]
    conn1 = synth.connectivity(8, 3, d * 3, seed=1)
    conn2 = synth.connectivity(4, 3, 8, seed=2)
    th1 = synth.table_logits(8, 8, seed=3)
    th2 = synth.table_logits(4, 8, seed=4)
    r = oracle.train_step(x, labels, thr, conn1, th1, conn2, th2, C, 1.5)

    def loss(t1, t2):
        return oracle.train_step(x, labels, thr, conn1, t1, conn2, t2, C, 1.5)["loss"]

    for which, (j, a) in [(1, (0, 0)), (1, (7, 5)), (2, (0, 3)), (2, (3, 7))]:
        base = th1 if which == 1 else th2
        tp, tm = base.copy(), base.copy()
        tp[j, a] = np.float32(base[j, a] + np.float32(1e-2))
        tm[j, a] = np.float32(base[j, a] - np.float32(1e-2))
        h = float(tp[j, a]) - float(tm[j, a])
        fd = ((loss(tp, th2) - loss(tm, th2)) if which == 1 else (loss(th1, tp) - loss(th1, tm))) / h
        got = r["dth1" if which == 1 else "dth2"][j, a]
        assert got == pytest.approx(fd, rel=1e-4, abs=1e-10)


# -------------------------------------------------------------------- hard --

def test_binarize_golden():
    rows = _gold_lines("binarize_edges.txt")
    th = np.array([float(r[0]) for r in rows], np.float32)
    want = [int(r[1]) for r in rows]
    th8 = np.zeros((len(th), 2), np.float32)
    th8[:, 1] = th                      # entry 1 of each node, entry 0 = 0.0
    tab = oracle.binarize_tables(th8)
    assert [(int(t) >> 1) & 1 for t in tab] == want
    assert all((int(t) & 1) == 0 for t in tab)


def _unpack(xp, N):
    bits = (xp[:, :, None] >> np.arange(32, dtype=np.uint32)[None, None, :]) & 1
    return bits.reshape(xp.shape[0], -1)[:, :N].astype(np.float64)


@pytest.mark.parametrize("N", [1, 31, 32, 33, 100])
def test_pack_is_encoder_packed(N):
    rng = np.random.default_rng(N)
    x = rng.integers(0, 256, size=(N, 6), dtype=np.uint8)
    thr = [32 * i for i in range(1, 8)]
    xp = oracle.pack_bits(x, thr)
    assert xp.shape == (42, (N + 31) // 32)
    np.testing.assert_array_equal(_unpack(xp, N), oracle.encode_thermometer(x, thr))
    # tail samples past N are zero
    if N % 32:
        assert np.all((xp[:, -1] >> np.uint32(N % 32)) == 0)


@pytest.mark.parametrize("k", [1, 2, 4, 6])
def test_hard_equals_soft_on_binarized(k):
    # correctness anchor of App. C.1: the bit-packed path equals the discrete
    # eager forward exactly for LightLUT; the soft node with tables at t in
    # {0, 1} (theta = +-800) on binary inputs is that discrete forward
    rng = np.random.default_rng(40 + k)
    w_in, w, N = 37, 23, 77
    Xb = rng.integers(0, 2, size=(w_in, N)).astype(np.float64)
    conn = synth.connectivity(w, k, w_in, seed=k)
    theta = synth.table_logits(w, 1 << k, seed=k + 1)
    th_hard = np.where(theta > 0, 800.0, -800.0).astype(np.float32)
    ysoft = oracle.lut_forward(Xb, conn, th_hard)
    assert set(np.unique(ysoft)) <= {0.0, 1.0}
    W = (N + 31) // 32
    xp = np.zeros((w_in, W), np.uint32)
    for s in range(N):
        xp[:, s // 32] |= (Xb[:, s].astype(np.uint32) << np.uint32(s % 32))
    yp = oracle.hard_forward(xp, N, conn, oracle.binarize_tables(theta))
    np.testing.assert_array_equal(_unpack(yp, N), ysoft)


def test_hard_brute_force_tiny():
    # independent per-sample lookup on python ints
    rng = np.random.default_rng(7)
    k, w_in, w, N = 3, 6, 4, 40
    bits = rng.integers(0, 2, size=(w_in, N))
    conn = synth.connectivity(w, k, w_in, seed=7)
    table = [int(v) for v in rng.integers(0, 256, size=w)]
    xp = np.zeros((w_in, 2), np.uint32)
    for r in range(w_in):
        for s in range(N):
            if bits[r, s]:
                xp[r, s // 32] |= np.uint32(1 << (s % 32))
    yp = oracle.hard_forward(xp, N, conn, np.array(table, np.uint64))
    for j in range(w):
        for s in range(N):
            a = sum(int(bits[conn[j, i], s]) << i for i in range(k))
            assert ((int(yp[j, s // 32]) >> (s % 32)) & 1) == ((table[j] >> a) & 1)


def test_popcount_head_golden():
    rows = _gold_lines("popcount_ties.txt")
    bits = np.array([[int(v) for v in r[1:]] for r in rows if r[0] == "bits"], np.uint32)
    N = bits.shape[1]
    yp = np.zeros((bits.shape[0], 1), np.uint32)
    for s in range(N):
        yp[:, 0] |= bits[:, s] << np.uint32(s)
    counts, pred = oracle.popcount_head(yp, N, 3)
    for r in rows:
        if r[0] == "sample":
            s = int(r[1])
            assert counts[s].tolist() == [int(v) for v in r[2:5]]
            assert pred[s] == int(r[5])


def test_popcount_head_random():
    rng = np.random.default_rng(8)
    C, g, N = 5, 7, 70
    yp = synth.random_words(C * g, 3, seed=8)
    counts, pred = oracle.popcount_head(yp, N, C)
    ub = _unpack(yp, N).reshape(C, g, N).sum(axis=1).T
    np.testing.assert_array_equal(counts, ub)
    np.testing.assert_array_equal(pred, np.argmax(ub, axis=1))


# ------------------------------------------------------------ generators --

def test_connectivity_unique_in_range():
    conn = synth.connectivity(5000, 6, 40, seed=3)
    assert conn.min() >= 0 and conn.max() < 40
    srt = np.sort(conn, axis=1)
    assert np.all(srt[:, 1:] != srt[:, :-1])


def test_blob_batch_shapes():
    x, lab = synth.blob_batch(300, 17, 4, 40.0, seed=1)
    assert x.dtype == torch.uint8 and x.shape == (300, 17)
    assert lab.dtype == torch.int32 and int(lab.min()) >= 0 and int(lab.max()) < 4
    x2, lab2 = synth.blob_batch(300, 17, 4, 40.0, seed=1)
    assert torch.equal(x, x2) and torch.equal(lab, lab2)


# ------------------------------------------------------------------ AdamW --

def test_adamw_matches_torch_optimizer():
    # the oracle's AdamW (§4 "Training") equals torch.optim.AdamW in float64
    # over several steps, with and without decoupled weight decay
    import torch
    rng = np.random.default_rng(11)
    for wd in (0.0, 0.05):
        theta0 = rng.standard_normal(300)
        p = torch.nn.Parameter(torch.tensor(theta0, dtype=torch.float64))
        opt = torch.optim.AdamW([p], lr=0.01, betas=(0.9, 0.999), eps=1e-8, weight_decay=wd)
        th, m, v = theta0.copy(), np.zeros(300), np.zeros(300)
        for t in range(1, 6):
            g = rng.standard_normal(300) * 10.0 ** rng.integers(-6, 1, size=300)
            p.grad = torch.tensor(g, dtype=torch.float64)
            opt.step()
            th, m, v = oracle.adamw_step(th, m, v, g, t, lr=0.01, wd=wd)
            st = opt.state[p]
            np.testing.assert_allclose(th, p.detach().numpy(), rtol=1e-12, atol=1e-15)
            np.testing.assert_allclose(m, st["exp_avg"].numpy(), rtol=1e-12, atol=0)
            np.testing.assert_allclose(v, st["exp_avg_sq"].numpy(), rtol=1e-12, atol=0)


def test_adamw_first_step_closed_form():
    # step 1 from zero moments: m = (1-b1) g, v = (1-b2) g^2, the bias
    # corrections cancel them, so theta moves by lr * g / (|g| + eps)
    rng = np.random.default_rng(12)
    theta0 = rng.standard_normal(50)
    g = rng.standard_normal(50) * 1e-3
    g[0] = 0.0
    th, m, v = oracle.adamw_step(theta0, np.zeros(50), np.zeros(50), g, 1, lr=0.01)
    np.testing.assert_allclose(m, 0.1 * g, rtol=1e-14, atol=0)      # (1 - 0.9) rounds in binary
    np.testing.assert_allclose(v, 0.001 * g * g, rtol=1e-14, atol=0)
    np.testing.assert_allclose(th, theta0 - 0.01 * g / (np.abs(g) + 1e-8), rtol=1e-12, atol=1e-15)
    assert th[0] == theta0[0]
    # zero gradient: only the decoupled decay moves theta
    th2, _, _ = oracle.adamw_step(theta0, np.zeros(50), np.zeros(50), np.zeros(50), 3, lr=0.01, wd=0.1)
    np.testing.assert_allclose(th2, theta0 * (1 - 0.01 * 0.1), rtol=1e-15, atol=0)
