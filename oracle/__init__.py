"""Python access to the CPU oracle (test infrastructure only).

Only ``tests/``, ``__graft_entry__.smoke()`` and the CPU-baseline leg of
``bench.py`` may import this package.  It loads ``liboracle.so`` built from
``bitlogic_oracle.c`` (plain C, double precision) and wraps each function for
numpy arrays.  It shares no code with the CUDA library.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "bitlogic_oracle.c")
_LIB = os.path.join(_HERE, "liboracle.so")
_lock = threading.Lock()
_lib = None


def build(force: bool = False) -> str:
    """Compile the oracle with gcc (OpenMP when available)."""
    if (not force and os.path.exists(_LIB)
            and os.path.getmtime(_LIB) >= os.path.getmtime(_SRC)):
        return _LIB
    tmp = _LIB + f".tmp{os.getpid()}"
    base = ["gcc", "-O2", "-std=c11", "-shared", "-fPIC", "-o", tmp, _SRC, "-lm"]
    try:
        subprocess.run(base[:1] + ["-fopenmp"] + base[1:], check=True,
                       capture_output=True)
    except subprocess.CalledProcessError:
        subprocess.run(base, check=True, capture_output=True)
    os.replace(tmp, _LIB)
    return _LIB


def _load():
    global _lib
    with _lock:
        if _lib is None:
            build()
            lib = ctypes.CDLL(_LIB)
            P = ctypes.c_void_p
            i32, i64, dbl = ctypes.c_int32, ctypes.c_int64, ctypes.c_double
            sig = {
                "oracle_max_threads": ([], ctypes.c_int),
                "oracle_set_threads": ([ctypes.c_int], None),
                "oracle_linear_thresholds": ([i32, P], None),
                "oracle_encode_thermometer": ([P, i64, i32, P, i32, P], None),
                "oracle_quantile_thresholds": ([P, i64, i32, P], None),
                "oracle_route_forward": ([P, i32, i64, P, P, i64, i32, P, P], None),
                "oracle_route_backward": ([P, i32, i64, P, P, i64, i32, P, P, P], None),
                "oracle_route_snap": ([P, P, i64, i32, P], None),
                "oracle_lut_forward": ([P, i32, i64, P, P, i32, i32, i32, P], None),
                "oracle_head_loss": ([P, i32, i64, i32, dbl, P, P, P, P], None),
                "oracle_lut_backward": ([P, i32, i64, P, P, i32, i32, i32, P, P, P], None),
                "oracle_binarize_tables": ([P, i32, i32, P], None),
                "oracle_pack_bits": ([P, i64, i32, P, i32, P], None),
                "oracle_hard_forward": ([P, i32, i64, P, P, i32, i32, P], None),
                "oracle_popcount_head": ([P, i32, i64, i32, P, P], None),
                "oracle_adamw_step": ([P, P, P, P, i64, i64, dbl, dbl, dbl, dbl, dbl], None),
            }
            for name, (args, res) in sig.items():
                fn = getattr(lib, name)
                fn.argtypes = args
                fn.restype = res
            _lib = lib
    return _lib


def _p(a):
    return None if a is None else a.ctypes.data_as(ctypes.c_void_p)


def _c(a, dtype):
    return np.ascontiguousarray(a, dtype=dtype)


def max_threads() -> int:
    return _load().oracle_max_threads()


def set_threads(n: int) -> None:
    _load().oracle_set_threads(int(n))


def linear_thresholds(b: int) -> np.ndarray:
    out = np.zeros(b, np.int32)
    _load().oracle_linear_thresholds(b, _p(out))
    return out


def encode_thermometer(x: np.ndarray, thr) -> np.ndarray:
    """x uint8 [B, d] -> bits float64 [d*b, B]."""
    x = _c(x, np.uint8)
    thr = _c(thr, np.uint8)
    B, d = x.shape
    bits = np.empty((d * thr.size, B), np.float64)
    _load().oracle_encode_thermometer(_p(x), B, d, _p(thr), thr.size, _p(bits))
    return bits


def quantile_thresholds(x: np.ndarray, b: int) -> np.ndarray:
    """Quantile thermometer thresholds (uint8 [b]) fitted on the flattened
    pixels of ``x`` (any shape, uint8, at least one value)."""
    x = _c(np.asarray(x).reshape(-1), np.uint8)
    if x.size == 0:
        raise ValueError("no pixels to fit")
    thr = np.empty(b, np.uint8)
    _load().oracle_quantile_thresholds(_p(x), x.size, int(b), _p(thr))
    return thr


NODES = {"soft": 0, "st": 1}


def _node(node: str) -> int:
    if node not in NODES:
        raise ValueError(f"node must be one of {sorted(NODES)}")
    return NODES[node]


def lut_forward(X: np.ndarray, conn: np.ndarray, theta: np.ndarray, node: str = "soft") -> np.ndarray:
    """X float64 [w_in, B], conn int32 [w, k], theta float32 [w, 2^k] -> Y float64 [w, B].
    node "soft": tables sigmoid(theta); "st": hard samples [theta > 0]
    (LightLUT straight-through)."""
    X = _c(X, np.float64)
    conn = _c(conn, np.int32)
    theta = _c(theta, np.float32)
    w_in, B = X.shape
    w, k = conn.shape
    assert theta.shape == (w, 1 << k)
    Y = np.empty((w, B), np.float64)
    _load().oracle_lut_forward(_p(X), w_in, B, _p(conn), _p(theta), w, k, _node(node), _p(Y))
    return Y


def head_loss(Y: np.ndarray, labels: np.ndarray, C: int, tau: float):
    """-> (logits float64 [B, C], loss float, dY float64 [w, B])."""
    Y = _c(Y, np.float64)
    labels = _c(labels, np.int32)
    w, B = Y.shape
    logits = np.empty((B, C), np.float64)
    dY = np.empty((w, B), np.float64)
    loss = np.zeros(1, np.float64)
    _load().oracle_head_loss(_p(Y), w, B, C, float(tau), _p(labels), _p(logits), _p(loss), _p(dY))
    return logits, float(loss[0]), dY


def lut_backward(X: np.ndarray, conn: np.ndarray, theta: np.ndarray, dY: np.ndarray,
                 want_dx: bool = True, node: str = "soft"):
    """-> (dtheta float64 [w, 2^k], dX float64 [w_in, B] or None).  node as
    in ``lut_forward``; for "st" dtheta is the straight-through estimate."""
    X = _c(X, np.float64)
    conn = _c(conn, np.int32)
    theta = _c(theta, np.float32)
    dY = _c(dY, np.float64)
    w_in, B = X.shape
    w, k = conn.shape
    dtheta = np.empty((w, 1 << k), np.float64)
    dX = np.empty((w_in, B), np.float64) if want_dx else None
    _load().oracle_lut_backward(_p(X), w_in, B, _p(conn), _p(theta), w, k, _node(node), _p(dY),
                                _p(dtheta), _p(dX))
    return dtheta, dX


def route_forward(X: np.ndarray, cand: np.ndarray, r: np.ndarray):
    """Learnable routing forward.  X float64 [w_in, B]; cand int32 [slots, Kc];
    r float32 [slots, Kc] -> (Xr float64 [slots, B], prob float64 [slots, Kc])."""
    X = _c(X, np.float64)
    cand = _c(cand, np.int32)
    r = _c(r, np.float32)
    w_in, B = X.shape
    n, Kc = cand.shape
    assert r.shape == (n, Kc) and Kc <= 64
    Xr = np.empty((n, B), np.float64)
    prob = np.empty((n, Kc), np.float64)
    _load().oracle_route_forward(_p(X), w_in, B, _p(cand), _p(r), n, Kc, _p(Xr), _p(prob))
    return Xr, prob


def route_backward(X: np.ndarray, cand: np.ndarray, r: np.ndarray, G: np.ndarray, want_dx: bool = True):
    """-> (dr float64 [slots, Kc], dX float64 [w_in, B] or None)."""
    X = _c(X, np.float64)
    cand = _c(cand, np.int32)
    r = _c(r, np.float32)
    G = _c(G, np.float64)
    w_in, B = X.shape
    n, Kc = cand.shape
    dr = np.empty((n, Kc), np.float64)
    dX = np.empty((w_in, B), np.float64) if want_dx else None
    _load().oracle_route_backward(_p(X), w_in, B, _p(cand), _p(r), n, Kc, _p(G), _p(dr), _p(dX))
    return dr, dX


def route_snap(cand: np.ndarray, r: np.ndarray) -> np.ndarray:
    """int32 [slots]: each slot's most likely candidate (first on ties)."""
    cand = _c(cand, np.int32)
    r = _c(r, np.float32)
    n, Kc = cand.shape
    conn = np.empty(n, np.int32)
    _load().oracle_route_snap(_p(cand), _p(r), n, Kc, _p(conn))
    return conn


def binarize_tables(theta: np.ndarray) -> np.ndarray:
    theta = _c(theta, np.float32)
    w, K = theta.shape
    k = K.bit_length() - 1
    table = np.empty(w, np.uint64)
    _load().oracle_binarize_tables(_p(theta), w, k, _p(table))
    return table


def pack_bits(x: np.ndarray, thr) -> np.ndarray:
    """x uint8 [N, d] -> xp uint32 [d*b, ceil(N/32)]."""
    x = _c(x, np.uint8)
    thr = _c(thr, np.uint8)
    N, d = x.shape
    xp = np.empty((d * thr.size, (N + 31) // 32), np.uint32)
    _load().oracle_pack_bits(_p(x), N, d, _p(thr), thr.size, _p(xp))
    return xp


def hard_forward(xp: np.ndarray, N: int, conn: np.ndarray, table: np.ndarray) -> np.ndarray:
    xp = _c(xp, np.uint32)
    conn = _c(conn, np.int32)
    table = _c(table, np.uint64)
    w_in, W = xp.shape
    assert W == (N + 31) // 32
    w, k = conn.shape
    yp = np.empty((w, W), np.uint32)
    _load().oracle_hard_forward(_p(xp), w_in, N, _p(conn), _p(table), w, k, _p(yp))
    return yp


def popcount_head(yp: np.ndarray, N: int, C: int):
    """-> (counts int32 [N, C], pred int32 [N])."""
    yp = _c(yp, np.uint32)
    w, W = yp.shape
    counts = np.empty((N, C), np.int32)
    pred = np.empty(N, np.int32)
    _load().oracle_popcount_head(_p(yp), w, N, C, _p(counts), _p(pred))
    return counts, pred


def adamw_step(theta: np.ndarray, m: np.ndarray, v: np.ndarray, g: np.ndarray, t: int,
               lr: float = 0.01, beta1: float = 0.9, beta2: float = 0.999, eps: float = 1e-8,
               wd: float = 0.0):
    """One AdamW step (§4 "Training"); returns new (theta, m, v) in float64."""
    th = _c(theta, np.float64).copy()
    mm = _c(m, np.float64).copy()
    vv = _c(v, np.float64).copy()
    gg = _c(g, np.float64)
    _load().oracle_adamw_step(_p(th), _p(mm), _p(vv), _p(gg), th.size, int(t), float(lr),
                              float(beta1), float(beta2), float(eps), float(wd))
    return th, mm, vv


# ---- composites used by the parity tests and the CPU baseline ------------

def train_step(x: np.ndarray, labels: np.ndarray, thr, conn1, th1, conn2, th2,
               C: int, tau: float, want_dx1: bool = False, node: str = "soft"):
    """Encoder -> two LUT layers -> group-sum head + CE -> both backwards
    (both layers of the node form ``node``)."""
    bits = encode_thermometer(x, thr)
    y1 = lut_forward(bits, conn1, th1, node)
    y2 = lut_forward(y1, conn2, th2, node)
    logits, loss, dy2 = head_loss(y2, labels, C, tau)
    dth2, dy1 = lut_backward(y1, conn2, th2, dy2, want_dx=True, node=node)
    dth1, dbits = lut_backward(bits, conn1, th1, dy1, want_dx=want_dx1, node=node)
    return dict(bits=bits, y1=y1, y2=y2, logits=logits, loss=loss, dy2=dy2,
                dth2=dth2, dy1=dy1, dth1=dth1, dbits=dbits)


def routed_train_step(x: np.ndarray, labels: np.ndarray, thr, cand1, r1, th1, cand2, r2, th2,
                      C: int, tau: float, node: str = "soft"):
    """Encoder -> two routed LUT layers (routing, then the node over the
    slot inputs) -> group-sum head + CE -> both backwards, through the
    routing as well."""
    w1, k1 = th1.shape[0], int(np.log2(th1.shape[1]))
    w2, k2 = th2.shape[0], int(np.log2(th2.shape[1]))
    id1 = np.arange(w1 * k1, dtype=np.int32).reshape(w1, k1)
    id2 = np.arange(w2 * k2, dtype=np.int32).reshape(w2, k2)
    bits = encode_thermometer(x, thr)
    xr1, p1 = route_forward(bits, cand1, r1)
    y1 = lut_forward(xr1, id1, th1, node)
    xr2, p2 = route_forward(y1, cand2, r2)
    y2 = lut_forward(xr2, id2, th2, node)
    logits, loss, dy2 = head_loss(y2, labels, C, tau)
    dth2, dxr2 = lut_backward(xr2, id2, th2, dy2, want_dx=True, node=node)
    dr2, dy1 = route_backward(y1, cand2, r2, dxr2, want_dx=True)
    dth1, dxr1 = lut_backward(xr1, id1, th1, dy1, want_dx=True, node=node)
    dr1, _ = route_backward(bits, cand1, r1, dxr1, want_dx=False)
    return dict(bits=bits, xr1=xr1, y1=y1, xr2=xr2, y2=y2, logits=logits, loss=loss, dy2=dy2,
                dth2=dth2, dxr2=dxr2, dr2=dr2, dy1=dy1, dth1=dth1, dxr1=dxr1, dr1=dr1, p1=p1, p2=p2)


def hard_infer(x: np.ndarray, thr, conn1, table1, conn2, table2, C: int):
    """Encode + pack -> two hard layers -> popcount head + argmax."""
    N = x.shape[0]
    xp = pack_bits(x, thr)
    yp1 = hard_forward(xp, N, conn1, table1)
    yp2 = hard_forward(yp1, N, conn2, table2)
    counts, pred = popcount_head(yp2, N, C)
    return dict(xp=xp, yp1=yp1, yp2=yp2, counts=counts, pred=pred)
