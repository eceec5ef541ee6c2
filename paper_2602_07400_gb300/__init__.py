"""Python binding of libbitlogic, the GB300 (sm_103a) LUT-network hot path.

Each function has the name of the C entry point it calls (see
``include/bitlogic.h``) and only marshals arguments: it checks dtypes,
devices and shapes of torch tensors, passes their device pointers and the
current CUDA stream, and raises ``BitLogicError`` on a non-zero status.  All
arithmetic runs in the library's CUDA kernels; there is no other code path.
If the library is missing or fails to load, every call raises.

Layouts: raw samples ``x`` uint8 [B, d]; soft activations fp32
[features, B] (batch contiguous); connectivity int32 [w, k]; table logits
fp32 [w, 2^k]; hard tables int64 [w] holding uint64 bit patterns; packed
bits int32 [rows, ceil(N/32)] holding uint32 words.
"""
from __future__ import annotations

import ctypes
import os
from typing import Optional, Tuple

import numpy as np
import torch

from . import build as _build

__all__ = [
    "BitLogicError", "load", "bitlogic_encode_thermometer", "bitlogic_lut_forward",
    "bitlogic_lut_backward_workspace", "bitlogic_lut_backward", "bitlogic_lut_backward_edges",
    "bitlogic_csr_reduce", "bitlogic_lut_backward_ex", "bitlogic_head_loss_ex",
    "bitlogic_head_loss_workspace", "bitlogic_head_loss_noalloc", "bitlogic_lut_backward_through", "bitlogic_lut_backward_through_u8",
    "bitlogic_lut_backward_u8", "bitlogic_lut_forward_u8", "bitlogic_encode_thermometer_bitrows",
    "bitlogic_lut_forward_bitrows", "bitlogic_lut_backward_bitrows", "bitrow_words",
    "bitlogic_head_loss", "bitlogic_binarize_tables", "bitlogic_pack_bits",
    "bitlogic_hard_forward", "bitlogic_build_csr", "bitlogic_csr_positions", "bitlogic_degree_order",
    "bitlogic_device_error",
    "bitlogic_adamw_update", "bitlogic_route_forward", "bitlogic_route_backward", "bitlogic_route_snap",
    "bitlogic_route_forward_u8", "bitlogic_route_backward_u8", "bitlogic_encode_thermometer_u8",
    "bitlogic_encode_thermometer_both",
    "bitlogic_pixel_histogram", "bitlogic_quantile_thresholds", "bitlogic_lut_forward_node", "bitlogic_lut_backward_node", "NODE_FORMS",
    "bitlogic_status_string", "bitlogic_version", "LIB_PATH",
    "bitlogic_issue_probe", "bitlogic_issue_probe_blocks", "bitlogic_issue_probe_threads", "bitlogic_issue_probe_ops_per_iter", "PROBE_KINDS",
]

LIB_PATH = _build.LIB

# node forms (bitlogic_node_t): the soft LightLUT node and its
# straight-through hard form
NODE_FORMS = {"soft": 0, "st": 1}

# instruction kinds of the issue-throughput probe (bitlogic_probe_t)
PROBE_KINDS = {"lop3": 0, "imad": 1, "ffma": 2, "mux3": 3, "mix": 4}


def _node_code(node) -> int:
    if isinstance(node, str):
        if node not in NODE_FORMS:
            raise ValueError(f"node must be one of {sorted(NODE_FORMS)}")
        return NODE_FORMS[node]
    return int(node)


class BitLogicError(RuntimeError):
    def __init__(self, fn: str, code: int, text: str):
        super().__init__(f"{fn}: status {code} ({text})")
        self.code = code


_lib = None
_P, _I32, _I64, _F32, _SZ = (ctypes.c_void_p, ctypes.c_int32, ctypes.c_int64,
                             ctypes.c_float, ctypes.c_size_t)
_SIGS = {
    "bitlogic_encode_thermometer": ([_P, _I64, _I32, _P, _I32, _P, _P], ctypes.c_int),
    "bitlogic_lut_forward": ([_P, _I32, _I64, _P, _P, _I32, _I32, _P, _P], ctypes.c_int),
    "bitlogic_pixel_histogram": ([_P, _I64, _P, _P], ctypes.c_int),
    "bitlogic_route_forward": ([_P, _I32, _I64, _P, _P, _I32, _I32, _P, _P, _P], ctypes.c_int),
    "bitlogic_route_backward": ([_P, _I32, _I64, _P, _P, _I32, _I32, _P, _P, _P, _P, _P, _P, _P], ctypes.c_int),
    "bitlogic_route_snap": ([_P, _P, _I32, _I32, _P, _P], ctypes.c_int),
    "bitlogic_route_forward_u8": ([_P, _I32, _I64, _P, _P, _I32, _I32, _P, _P, _P], ctypes.c_int),
    "bitlogic_route_backward_u8": ([_P, _I32, _I64, _P, _P, _I32, _I32, _P, _P, _P], ctypes.c_int),
    "bitlogic_encode_thermometer_u8": ([_P, _I64, _I32, _P, _I32, _P, _P], ctypes.c_int),
    "bitlogic_encode_thermometer_both": ([_P, _I64, _I32, _P, _I32, _P, _P, _P], ctypes.c_int),
    "bitlogic_quantile_thresholds": ([_P, _I32, _P], ctypes.c_int),
    "bitlogic_lut_forward_node": ([_P, _I32, _I64, _P, _P, _I32, _I32, _I32, _P, _P], ctypes.c_int),
    "bitlogic_lut_forward_u8": ([_P, _I32, _I64, _P, _P, _I32, _I32, _I32, _P, _P], ctypes.c_int),
    "bitlogic_encode_thermometer_bitrows": ([_P, _I64, _I32, _P, _I32, _P, _P], ctypes.c_int),
    "bitlogic_lut_forward_bitrows": ([_P, _I32, _I64, _P, _P, _I32, _I32, _I32, _P, _P], ctypes.c_int),
    "bitlogic_lut_backward_bitrows": ([_P, _I32, _I64, _P, _P, _I32, _I32, _I32, _P, _I32, _P, _P, _P, _I32, _P,
                                       _P, _P, _P], ctypes.c_int),
    "bitlogic_degree_order": ([_P, _I32, _P], ctypes.c_int),
    "bitlogic_lut_backward_workspace": ([_I32, _I64, _I32, _I32, _I32], _SZ),
    "bitlogic_lut_backward": ([_P, _I32, _I64, _P, _P, _I32, _I32, _P, _P, _P, _P, _P,
                               _P, _SZ, _P], ctypes.c_int),
    "bitlogic_lut_backward_edges": ([_P, _I32, _I64, _P, _P, _I32, _I32, _P, _P, _P, _P],
                                    ctypes.c_int),
    "bitlogic_csr_reduce": ([_P, _I64, _P, _P, _I32, _I32, _P, _P], ctypes.c_int),
    "bitlogic_lut_backward_ex": ([_P, _I32, _I64, _P, _P, _I32, _I32, _P, _I32, _P, _P, _P, _I32,
                                  _P, _P, _P, _P, _P], ctypes.c_int),
    "bitlogic_lut_backward_node": ([_P, _I32, _I64, _P, _P, _I32, _I32, _I32, _P, _I32, _P, _P, _P, _I32,
                                    _P, _P, _P, _P, _P], ctypes.c_int),
    "bitlogic_lut_backward_through": ([_P, _I32, _I64, _P, _P, _I32, _I32, _I32, _P, _P, _P, _I32, _I32, _P, _I32,
                                       _P, _P, _P, _P, _P], ctypes.c_int),
    "bitlogic_lut_backward_through_u8": ([_P, _I32, _I64, _P, _P, _I32, _I32, _I32, _P, _P, _P, _I32, _I32, _P,
                                          _I32, _P, _P, _P, _P, _P], ctypes.c_int),
    "bitlogic_lut_backward_u8": ([_P, _I32, _I64, _P, _P, _I32, _I32, _I32, _P, _I32, _P, _P, _P, _I32, _P, _P, _P],
                                 ctypes.c_int),
    "bitlogic_head_loss_ex": ([_P, _I32, _I64, _I32, _F32, _P, _P, _P, _P, _P, _P, _SZ, _P],
                              ctypes.c_int),
    "bitlogic_head_loss_workspace": ([_I64, _I32], _SZ),
    "bitlogic_head_loss_noalloc": ([_P, _I32, _I64, _I32, _F32, _P, _P, _P, _P, _P], ctypes.c_int),
    "bitlogic_head_loss": ([_P, _I32, _I64, _I32, _F32, _P, _P, _P, _P, _P, _SZ, _P],
                           ctypes.c_int),
    "bitlogic_binarize_tables": ([_P, _I32, _I32, _P, _P], ctypes.c_int),
    "bitlogic_pack_bits": ([_P, _I64, _I32, _P, _I32, _P, _P], ctypes.c_int),
    "bitlogic_hard_forward": ([_P, _I32, _I64, _P, _P, _I32, _I32, _P, _I32, _P, _P, _P],
                              ctypes.c_int),
    "bitlogic_build_csr": ([_P, _I32, _I32, _I32, _P, _P], ctypes.c_int),
    "bitlogic_csr_positions": ([_P, _I32, _P], ctypes.c_int),
    "bitlogic_adamw_update": ([_P, _P, _P, _P, _I64, _I64, _F32, _F32, _F32, _F32, _F32, _P], ctypes.c_int),
    "bitlogic_device_error": ([_P], ctypes.c_int),
    "bitlogic_status_string": ([ctypes.c_int], ctypes.c_char_p),
    "bitlogic_version": ([], ctypes.c_int),
    "bitlogic_issue_probe_blocks": ([], _I64),
    "bitlogic_issue_probe_threads": ([], _I64),
    "bitlogic_issue_probe_ops_per_iter": ([], _I64),
    "bitlogic_issue_probe": ([_I32, _I64, ctypes.c_uint32, _P, _I64, _P, _P], ctypes.c_int),
}


def load(build_if_missing: bool = True):
    """Load (building first if needed) the CUDA library; raises if absent."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH) or not _build.up_to_date():
            if not build_if_missing:
                raise RuntimeError(f"CUDA library {LIB_PATH} is missing")
            _build.build()
        lib = ctypes.CDLL(LIB_PATH)
        for name, (args, res) in _SIGS.items():
            fn = getattr(lib, name)
            fn.argtypes = args
            fn.restype = res
        _lib = lib
    return _lib


def _check(fn: str, code: int):
    if code != 0:
        raise BitLogicError(fn, code, bitlogic_status_string(code))


def _ptr(t: Optional[torch.Tensor]):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


def _stream(stream) -> ctypes.c_void_p:
    if stream is None:
        stream = torch.cuda.current_stream()
    return ctypes.c_void_p(stream.cuda_stream)


def _need(t: torch.Tensor, name: str, dtype: torch.dtype, shape: Tuple[int, ...]):
    if not isinstance(t, torch.Tensor):
        raise TypeError(f"{name} must be a torch.Tensor")
    if t.dtype != dtype:
        raise TypeError(f"{name}: expected {dtype}, got {t.dtype}")
    if not t.is_cuda:
        raise ValueError(f"{name} must be on a CUDA device")
    if not t.is_contiguous():
        raise ValueError(f"{name} must be contiguous")
    if tuple(t.shape) != tuple(shape):
        raise ValueError(f"{name}: expected shape {tuple(shape)}, got {tuple(t.shape)}")


def _thr_buf(thresholds) -> Tuple[ctypes.Array, int]:
    vals = [int(v) for v in thresholds]
    if any(v < 0 or v > 255 for v in vals):
        raise ValueError("thresholds must be uint8 values")
    return (ctypes.c_uint8 * max(1, len(vals)))(*vals), len(vals)


def bitlogic_status_string(code: int) -> str:
    return load().bitlogic_status_string(int(code)).decode()


def bitlogic_version() -> int:
    return load().bitlogic_version()


def bitlogic_issue_probe_blocks() -> int:
    return int(load().bitlogic_issue_probe_blocks())


def bitlogic_issue_probe_threads() -> int:
    return int(load().bitlogic_issue_probe_threads())


def bitlogic_issue_probe_ops_per_iter() -> int:
    return int(load().bitlogic_issue_probe_ops_per_iter())


def bitlogic_issue_probe(kind, iters: int, sink: torch.Tensor, cycles: Optional[torch.Tensor] = None,
                         seed: int = 1, stream=None):
    """One launch of the issue-throughput probe: bitlogic_issue_probe_threads()
    threads x iters x bitlogic_issue_probe_ops_per_iter() instructions of
    `kind` ("lop3", "imad", "ffma", "mux3" or "mix"); `cycles` (int64 CUDA
    tensor of bitlogic_issue_probe_blocks() entries, optional) receives the
    SM clock cycles of each block."""
    if isinstance(kind, str):
        if kind not in PROBE_KINDS:
            raise ValueError(f"kind must be one of {sorted(PROBE_KINDS)}")
        kind = PROBE_KINDS[kind]
    if not isinstance(sink, torch.Tensor) or sink.dtype != torch.int32 or not sink.is_cuda \
            or not sink.is_contiguous():
        raise ValueError("sink must be a contiguous int32 CUDA tensor")
    if cycles is not None:
        _need(cycles, "cycles", torch.int64, (bitlogic_issue_probe_blocks(),))
    _check("bitlogic_issue_probe", load().bitlogic_issue_probe(
        int(kind), int(iters), int(seed) & 0xffffffff, _ptr(sink), sink.numel(), _ptr(cycles), _stream(stream)))


def bitlogic_encode_thermometer(x: torch.Tensor, thresholds, bits: torch.Tensor, stream=None):
    B, d = x.shape
    buf, b = _thr_buf(thresholds)
    _need(x, "x", torch.uint8, (B, d))
    _need(bits, "bits", torch.float32, (d * b, B))
    _check("bitlogic_encode_thermometer", load().bitlogic_encode_thermometer(
        _ptr(x), B, d, buf, b, _ptr(bits), _stream(stream)))


def bitlogic_encode_thermometer_u8(x: torch.Tensor, thresholds, bits: torch.Tensor, stream=None):
    B, d = x.shape
    buf, b = _thr_buf(thresholds)
    _need(x, "x", torch.uint8, (B, d))
    _need(bits, "bits", torch.uint8, (d * b, B))
    _check("bitlogic_encode_thermometer_u8", load().bitlogic_encode_thermometer_u8(
        _ptr(x), B, d, buf, b, _ptr(bits), _stream(stream)))


def bitrow_words(B: int) -> int:
    """32-bit words per wire bit row of a batch of B (32 per 1024-sample block)."""
    return 32 * ((int(B) + 1023) // 1024)


def bitlogic_encode_thermometer_bitrows(x: torch.Tensor, thresholds, bits: torch.Tensor, stream=None):
    """The thermometer wires at one bit per sample, [d*b, bitrow_words(B)] int32."""
    B, d = x.shape
    buf, b = _thr_buf(thresholds)
    _need(x, "x", torch.uint8, (B, d))
    _need(bits, "bits", torch.int32, (d * b, bitrow_words(B)))
    _check("bitlogic_encode_thermometer_bitrows", load().bitlogic_encode_thermometer_bitrows(
        _ptr(x), B, d, buf, b, _ptr(bits), _stream(stream)))


def bitlogic_encode_thermometer_both(x: torch.Tensor, thresholds, bits: torch.Tensor, bits8: torch.Tensor,
                                     stream=None):
    """The thermometer wires as fp32 rows and as byte rows, in one pass."""
    B, d = x.shape
    thr, b = _thr_buf(thresholds)
    _need(x, "x", torch.uint8, (B, d))
    _need(bits, "bits", torch.float32, (d * b, B))
    _need(bits8, "bits8", torch.uint8, (d * b, B))
    _check("bitlogic_encode_thermometer_both", load().bitlogic_encode_thermometer_both(
        _ptr(x), B, d, thr, b, _ptr(bits), _ptr(bits8), _stream(stream)))


def bitlogic_route_forward_u8(X: torch.Tensor, cand: torch.Tensor, r: torch.Tensor, Xr: torch.Tensor,
                              prob: Optional[torch.Tensor] = None, stream=None):
    """bitlogic_route_forward over a uint8 layer input [w_in, B]."""
    _route_forward("bitlogic_route_forward_u8", torch.uint8, X, cand, r, Xr, prob, stream)


def bitlogic_route_backward_u8(X: torch.Tensor, cand: torch.Tensor, r: torch.Tensor, G: torch.Tensor,
                               dr: torch.Tensor, stream=None):
    """dr of a routing over a uint8 layer input (no input gradient)."""
    w_in, B = X.shape
    slots, Kc = cand.shape
    _need(X, "X", torch.uint8, (w_in, B))
    _need(cand, "cand", torch.int32, (slots, Kc))
    _need(r, "r", torch.float32, (slots, Kc))
    _need(G, "G", torch.float32, (slots, B))
    _need(dr, "dr", torch.float32, (slots, Kc))
    _check("bitlogic_route_backward_u8", load().bitlogic_route_backward_u8(
        _ptr(X), w_in, B, _ptr(cand), _ptr(r), slots, Kc, _ptr(G), _ptr(dr), _stream(stream)))


def bitlogic_route_forward(X: torch.Tensor, cand: torch.Tensor, r: torch.Tensor, Xr: torch.Tensor,
                           prob: Optional[torch.Tensor] = None, stream=None):
    """Slot inputs of learnable routing: cand int32 [slots, Kc], r fp32
    [slots, Kc] -> Xr fp32 [slots, B] (and the probabilities into prob)."""
    _route_forward("bitlogic_route_forward", torch.float32, X, cand, r, Xr, prob, stream)


def _route_forward(fn, dtype, X, cand, r, Xr, prob, stream):
    w_in, B = X.shape
    slots, Kc = cand.shape
    _need(X, "X", dtype, (w_in, B))
    _need(cand, "cand", torch.int32, (slots, Kc))
    _need(r, "r", torch.float32, (slots, Kc))
    _need(Xr, "Xr", torch.float32, (slots, B))
    if prob is not None:
        _need(prob, "prob", torch.float32, (slots, Kc))
    _check(fn, getattr(load(), fn)(
        _ptr(X), w_in, B, _ptr(cand), _ptr(r), slots, Kc, _ptr(Xr), _ptr(prob), _stream(stream)))


def bitlogic_route_backward(X: torch.Tensor, cand: torch.Tensor, r: torch.Tensor, G: torch.Tensor,
                            dr: torch.Tensor, prob: Optional[torch.Tensor] = None,
                            csr_off: Optional[torch.Tensor] = None, csr_edge: Optional[torch.Tensor] = None,
                            dX: Optional[torch.Tensor] = None, stream=None):
    """dr from the slot-input gradient G; dX (with prob and the candidate
    CSR map) when given."""
    w_in, B = X.shape
    slots, Kc = cand.shape
    _need(X, "X", torch.float32, (w_in, B))
    _need(cand, "cand", torch.int32, (slots, Kc))
    _need(r, "r", torch.float32, (slots, Kc))
    _need(G, "G", torch.float32, (slots, B))
    _need(dr, "dr", torch.float32, (slots, Kc))
    if dX is not None:
        _need(dX, "dX", torch.float32, (w_in, B))
        _need(prob, "prob", torch.float32, (slots, Kc))
        _need(csr_off, "csr_off", torch.int32, (w_in + 1,))
        _need(csr_edge, "csr_edge", torch.int32, (slots * Kc,))
    _check("bitlogic_route_backward", load().bitlogic_route_backward(
        _ptr(X), w_in, B, _ptr(cand), _ptr(r), slots, Kc, _ptr(G), _ptr(dr), _ptr(prob), _ptr(csr_off),
        _ptr(csr_edge), _ptr(dX), _stream(stream)))


def bitlogic_route_snap(cand: torch.Tensor, r: torch.Tensor, conn: torch.Tensor, stream=None):
    """conn int32 [slots]: each slot's most likely candidate (first on ties)."""
    slots, Kc = cand.shape
    _need(cand, "cand", torch.int32, (slots, Kc))
    _need(r, "r", torch.float32, (slots, Kc))
    _need(conn, "conn", torch.int32, (slots,))
    _check("bitlogic_route_snap", load().bitlogic_route_snap(
        _ptr(cand), _ptr(r), slots, Kc, _ptr(conn), _stream(stream)))


def bitlogic_pixel_histogram(x: torch.Tensor, hist: torch.Tensor, stream=None):
    """hist (int64 [256] on the device, holding uint64 counts) += the value
    counts of the bytes of x (uint8, any shape, contiguous)."""
    if not isinstance(x, torch.Tensor) or x.dtype != torch.uint8 or not x.is_cuda or not x.is_contiguous():
        raise TypeError("x must be a contiguous uint8 CUDA tensor")
    _need(hist, "hist", torch.int64, (256,))
    _check("bitlogic_pixel_histogram", load().bitlogic_pixel_histogram(
        _ptr(x), x.numel(), _ptr(hist), _stream(stream)))


def bitlogic_quantile_thresholds(hist, b: int) -> np.ndarray:
    """Quantile thermometer thresholds (uint8 [b]) from a finished
    histogram (256 counts, host array or tensor)."""
    if isinstance(hist, torch.Tensor):
        hist = hist.detach().cpu().numpy()
    h = np.ascontiguousarray(np.asarray(hist).astype(np.uint64))
    if h.shape != (256,):
        raise ValueError("hist must hold 256 counts")
    thr = np.empty(max(1, int(b)), np.uint8)
    _check("bitlogic_quantile_thresholds", load().bitlogic_quantile_thresholds(
        h.ctypes.data_as(ctypes.c_void_p), int(b), thr.ctypes.data_as(ctypes.c_void_p)))
    return thr[:b]


def bitlogic_lut_forward(X: torch.Tensor, conn: torch.Tensor, theta: torch.Tensor,
                         Y: torch.Tensor, stream=None):
    w_in, B = X.shape
    w, k = conn.shape
    _need(X, "X", torch.float32, (w_in, B))
    _need(conn, "conn", torch.int32, (w, k))
    _need(theta, "theta", torch.float32, (w, 1 << k))
    _need(Y, "Y", torch.float32, (w, B))
    _check("bitlogic_lut_forward", load().bitlogic_lut_forward(
        _ptr(X), w_in, B, _ptr(conn), _ptr(theta), w, k, _ptr(Y), _stream(stream)))


def bitlogic_lut_forward_node(X: torch.Tensor, conn: torch.Tensor, theta: torch.Tensor,
                              Y: torch.Tensor, node="soft", stream=None):
    """node "soft" or "st" (or the bitlogic_node_t value)."""
    code = _node_code(node)
    w_in, B = X.shape
    w, k = conn.shape
    _need(X, "X", torch.float32, (w_in, B))
    _need(conn, "conn", torch.int32, (w, k))
    _need(theta, "theta", torch.float32, (w, 1 << k))
    _need(Y, "Y", torch.float32, (w, B))
    _check("bitlogic_lut_forward_node", load().bitlogic_lut_forward_node(
        _ptr(X), w_in, B, _ptr(conn), _ptr(theta), w, k, code, _ptr(Y), _stream(stream)))


def bitlogic_lut_forward_u8(X: torch.Tensor, conn: torch.Tensor, theta: torch.Tensor,
                            Y: torch.Tensor, node="soft", stream=None):
    """Layer forward on byte rows (binary wires): Y[j][s] = the table entry
    the inputs' bits select."""
    code = _node_code(node)
    w_in, B = X.shape
    w, k = conn.shape
    _need(X, "X", torch.uint8, (w_in, B))
    _need(conn, "conn", torch.int32, (w, k))
    _need(theta, "theta", torch.float32, (w, 1 << k))
    _need(Y, "Y", torch.float32, (w, B))
    _check("bitlogic_lut_forward_u8", load().bitlogic_lut_forward_u8(
        _ptr(X), w_in, B, _ptr(conn), _ptr(theta), w, k, code, _ptr(Y), _stream(stream)))


def bitlogic_lut_forward_bitrows(X: torch.Tensor, B: int, conn: torch.Tensor, theta: torch.Tensor,
                                 Y: torch.Tensor, node="soft", stream=None):
    """Layer forward on wire bit rows X [w_in, bitrow_words(B)] int32 (binary
    wires at one bit per sample): the table entry the inputs' bits select."""
    code = _node_code(node)
    w_in = X.shape[0]
    w, k = conn.shape
    _need(X, "X", torch.int32, (w_in, bitrow_words(B)))
    _need(conn, "conn", torch.int32, (w, k))
    _need(theta, "theta", torch.float32, (w, 1 << k))
    _need(Y, "Y", torch.float32, (w, B))
    _check("bitlogic_lut_forward_bitrows", load().bitlogic_lut_forward_bitrows(
        _ptr(X), w_in, B, _ptr(conn), _ptr(theta), w, k, code, _ptr(Y), _stream(stream)))


def bitlogic_lut_backward_workspace(w_in: int, B: int, w: int, k: int, want_dx: bool) -> int:
    return int(load().bitlogic_lut_backward_workspace(w_in, B, w, k, int(bool(want_dx))))


def bitlogic_lut_backward(X: torch.Tensor, conn: torch.Tensor, theta: torch.Tensor,
                          dY: torch.Tensor, dtheta: torch.Tensor,
                          dX: Optional[torch.Tensor] = None,
                          csr_off: Optional[torch.Tensor] = None,
                          csr_edge: Optional[torch.Tensor] = None,
                          workspace: Optional[torch.Tensor] = None, stream=None):
    w_in, B = X.shape
    w, k = conn.shape
    _need(X, "X", torch.float32, (w_in, B))
    _need(conn, "conn", torch.int32, (w, k))
    _need(theta, "theta", torch.float32, (w, 1 << k))
    _need(dY, "dY", torch.float32, (w, B))
    _need(dtheta, "dtheta", torch.float32, (w, 1 << k))
    ws_bytes = 0
    if dX is not None:
        _need(dX, "dX", torch.float32, (w_in, B))
        _need(csr_off, "csr_off", torch.int32, (w_in + 1,))
        _need(csr_edge, "csr_edge", torch.int32, (w * k,))
        if workspace is None or not workspace.is_cuda or workspace.dtype != torch.uint8:
            raise ValueError("workspace: uint8 CUDA tensor required when dX is requested")
        ws_bytes = workspace.numel()
    _check("bitlogic_lut_backward", load().bitlogic_lut_backward(
        _ptr(X), w_in, B, _ptr(conn), _ptr(theta), w, k, _ptr(dY), _ptr(csr_off),
        _ptr(csr_edge), _ptr(dtheta), _ptr(dX), _ptr(workspace), ws_bytes, _stream(stream)))


def bitlogic_lut_backward_edges(X: torch.Tensor, conn: torch.Tensor, theta: torch.Tensor,
                                dY: torch.Tensor, dtheta: torch.Tensor,
                                edge_terms: Optional[torch.Tensor] = None, stream=None):
    w_in, B = X.shape
    w, k = conn.shape
    _need(X, "X", torch.float32, (w_in, B))
    _need(conn, "conn", torch.int32, (w, k))
    _need(theta, "theta", torch.float32, (w, 1 << k))
    _need(dY, "dY", torch.float32, (w, B))
    _need(dtheta, "dtheta", torch.float32, (w, 1 << k))
    if edge_terms is not None:
        _need(edge_terms, "edge_terms", torch.float32, (w * k, B))
    _check("bitlogic_lut_backward_edges", load().bitlogic_lut_backward_edges(
        _ptr(X), w_in, B, _ptr(conn), _ptr(theta), w, k, _ptr(dY), _ptr(dtheta),
        _ptr(edge_terms), _stream(stream)))


def bitlogic_csr_reduce(edge_terms: torch.Tensor, csr_off: torch.Tensor,
                        csr_edge: Optional[torch.Tensor], dX: torch.Tensor, stream=None):
    """csr_edge None: the term rows are stored in CSR order."""
    nE, B = edge_terms.shape
    w_in = dX.shape[0]
    _need(edge_terms, "edge_terms", torch.float32, (nE, B))
    _need(csr_off, "csr_off", torch.int32, (w_in + 1,))
    if csr_edge is not None:
        _need(csr_edge, "csr_edge", torch.int32, (nE,))
    _need(dX, "dX", torch.float32, (w_in, B))
    _check("bitlogic_csr_reduce", load().bitlogic_csr_reduce(
        _ptr(edge_terms), B, _ptr(csr_off), _ptr(csr_edge), w_in, nE, _ptr(dX), _stream(stream)))


def bitlogic_lut_backward_ex(X: torch.Tensor, conn: torch.Tensor, theta: torch.Tensor,
                             dtheta: torch.Tensor, dY: Optional[torch.Tensor] = None,
                             dy_group: int = 1, up_terms: Optional[torch.Tensor] = None,
                             up_off: Optional[torch.Tensor] = None,
                             up_edge: Optional[torch.Tensor] = None,
                             edge_terms: Optional[torch.Tensor] = None,
                             edge_pos: Optional[torch.Tensor] = None,
                             dY_out: Optional[torch.Tensor] = None, stream=None):
    """up_edge None with up_terms: the upstream term rows are in CSR order.
    edge_pos: store the term of edge e at row edge_pos[e] of edge_terms."""
    _backward_general("bitlogic_lut_backward_ex", None, X, conn, theta, dtheta, dY, dy_group, up_terms,
                      up_off, up_edge, edge_terms, edge_pos, dY_out, stream)


def bitlogic_lut_backward_node(X: torch.Tensor, conn: torch.Tensor, theta: torch.Tensor,
                               dtheta: torch.Tensor, node="soft", dY: Optional[torch.Tensor] = None,
                               dy_group: int = 1, up_terms: Optional[torch.Tensor] = None,
                               up_off: Optional[torch.Tensor] = None,
                               up_edge: Optional[torch.Tensor] = None,
                               edge_terms: Optional[torch.Tensor] = None,
                               edge_pos: Optional[torch.Tensor] = None,
                               dY_out: Optional[torch.Tensor] = None, stream=None):
    """bitlogic_lut_backward_ex for the node form ``node`` ("soft" or "st")."""
    _backward_general("bitlogic_lut_backward_node", _node_code(node), X, conn, theta, dtheta, dY, dy_group,
                      up_terms, up_off, up_edge, edge_terms, edge_pos, dY_out, stream)


def _backward_general(fn, node, X, conn, theta, dtheta, dY, dy_group, up_terms, up_off, up_edge,
                      edge_terms, edge_pos, dY_out, stream):
    w_in, B = X.shape
    w, k = conn.shape
    _need(X, "X", torch.float32, (w_in, B))
    _need(conn, "conn", torch.int32, (w, k))
    _need(theta, "theta", torch.float32, (w, 1 << k))
    _need(dtheta, "dtheta", torch.float32, (w, 1 << k))
    n_up = 0
    if dY is not None:
        if w % dy_group != 0:
            raise ValueError("dy_group must divide w")
        _need(dY, "dY", torch.float32, (w // dy_group, B))
    if up_terms is not None:
        n_up = up_terms.shape[0]
        _need(up_terms, "up_terms", torch.float32, (n_up, B))
        _need(up_off, "up_off", torch.int32, (w + 1,))
        if up_edge is not None:
            _need(up_edge, "up_edge", torch.int32, (n_up,))
    if edge_terms is not None:
        _need(edge_terms, "edge_terms", torch.float32, (w * k, B))
    if edge_pos is not None:
        _need(edge_pos, "edge_pos", torch.int32, (w * k,))
    if dY_out is not None:
        _need(dY_out, "dY_out", torch.float32, (w, B))
    rest = (_ptr(dY), int(dy_group), _ptr(up_terms), _ptr(up_off), _ptr(up_edge), n_up, _ptr(dtheta),
            _ptr(edge_terms), _ptr(edge_pos), _ptr(dY_out), _stream(stream))
    head = (_ptr(X), w_in, B, _ptr(conn), _ptr(theta), w, k)
    args = head + rest if node is None else head + (node,) + rest
    _check(fn, getattr(load(), fn)(*args))


def bitlogic_lut_backward_through(X: torch.Tensor, conn: torch.Tensor, theta: torch.Tensor, dtheta: torch.Tensor,
                                  Y: torch.Tensor, up_conn: torch.Tensor, up_theta: torch.Tensor,
                                  up_dY: torch.Tensor, up_group: int, up_off: torch.Tensor,
                                  up_edge: Optional[torch.Tensor] = None, node="soft",
                                  dY_out: Optional[torch.Tensor] = None, stream=None):
    """Table gradient of a layer from the next layer's output gradient,
    recomputing this layer's output gradient through the next layer (fan-in
    1..3) instead of reading stored per-edge terms.  X: fp32 rows, or uint8
    rows of binary wires."""
    w_in, B = X.shape
    w, k = conn.shape
    up_w, up_k = up_conn.shape
    if X.dtype == torch.uint8:
        _need(X, "X", torch.uint8, (w_in, B))
        fn = "bitlogic_lut_backward_through_u8"
    else:
        _need(X, "X", torch.float32, (w_in, B))
        fn = "bitlogic_lut_backward_through"
    _need(conn, "conn", torch.int32, (w, k))
    _need(theta, "theta", torch.float32, (w, 1 << k))
    _need(dtheta, "dtheta", torch.float32, (w, 1 << k))
    _need(Y, "Y", torch.float32, (w, B))
    _need(up_conn, "up_conn", torch.int32, (up_w, up_k))
    _need(up_theta, "up_theta", torch.float32, (up_w, 1 << up_k))
    if up_group < 1 or up_w % up_group != 0:
        raise ValueError("up_group must divide the next layer's width")
    _need(up_dY, "up_dY", torch.float32, (up_w // up_group, B))
    _need(up_off, "up_off", torch.int32, (w + 1,))
    if up_edge is not None:
        _need(up_edge, "up_edge", torch.int32, (up_w * up_k,))
    if dY_out is not None:
        _need(dY_out, "dY_out", torch.float32, (w, B))
    _check(fn, getattr(load(), fn)(
        _ptr(X), w_in, B, _ptr(conn), _ptr(theta), w, k, _node_code(node), _ptr(Y), _ptr(up_conn),
        _ptr(up_theta), up_w, up_k, _ptr(up_dY), int(up_group), _ptr(up_off), _ptr(up_edge), _ptr(dtheta),
        _ptr(dY_out), _stream(stream)))


def bitlogic_lut_backward_through_u8(X: torch.Tensor, *args, **kwargs):
    """bitlogic_lut_backward_through with X as uint8 rows of binary wires."""
    if not isinstance(X, torch.Tensor) or X.dtype != torch.uint8:
        raise TypeError("X must be a uint8 tensor")
    bitlogic_lut_backward_through(X, *args, **kwargs)


def bitlogic_lut_backward_u8(X: torch.Tensor, conn: torch.Tensor, theta: torch.Tensor, dtheta: torch.Tensor,
                             node="soft", dY: Optional[torch.Tensor] = None, dy_group: int = 1,
                             up_terms: Optional[torch.Tensor] = None, up_off: Optional[torch.Tensor] = None,
                             up_edge: Optional[torch.Tensor] = None, dY_out: Optional[torch.Tensor] = None,
                             stream=None):
    """Table gradient of a layer whose input is byte rows (binary wires),
    from dY rows or from the next layer's per-edge terms (no input gradient)."""
    w_in, B = X.shape
    w, k = conn.shape
    _need(X, "X", torch.uint8, (w_in, B))
    _need(conn, "conn", torch.int32, (w, k))
    _need(theta, "theta", torch.float32, (w, 1 << k))
    _need(dtheta, "dtheta", torch.float32, (w, 1 << k))
    n_up = 0
    if dY is not None:
        if w % dy_group != 0:
            raise ValueError("dy_group must divide w")
        _need(dY, "dY", torch.float32, (w // dy_group, B))
    if up_terms is not None:
        n_up = up_terms.shape[0]
        _need(up_terms, "up_terms", torch.float32, (n_up, B))
        _need(up_off, "up_off", torch.int32, (w + 1,))
        if up_edge is not None:
            _need(up_edge, "up_edge", torch.int32, (n_up,))
    if dY_out is not None:
        _need(dY_out, "dY_out", torch.float32, (w, B))
    _check("bitlogic_lut_backward_u8", load().bitlogic_lut_backward_u8(
        _ptr(X), w_in, B, _ptr(conn), _ptr(theta), w, k, _node_code(node), _ptr(dY), int(dy_group),
        _ptr(up_terms), _ptr(up_off), _ptr(up_edge), n_up, _ptr(dtheta), _ptr(dY_out), _stream(stream)))


def bitlogic_lut_backward_bitrows(X: torch.Tensor, B: int, conn: torch.Tensor, theta: torch.Tensor,
                                  dtheta: torch.Tensor, node="soft", dY: Optional[torch.Tensor] = None,
                                  dy_group: int = 1, up_terms: Optional[torch.Tensor] = None,
                                  up_off: Optional[torch.Tensor] = None, up_edge: Optional[torch.Tensor] = None,
                                  dY_out: Optional[torch.Tensor] = None, order: Optional[torch.Tensor] = None,
                                  stream=None):
    """bitlogic_lut_backward_u8 on wire bit rows X [w_in, bitrow_words(B)] int32;
    ``order`` (int32 [w], e.g. bitlogic_degree_order(up_off)) is the order
    in which the nodes are taken (no effect on the results)."""
    w_in = X.shape[0]
    _need(X, "X", torch.int32, (w_in, bitrow_words(B)))
    w, k = conn.shape
    _need(conn, "conn", torch.int32, (w, k))
    _need(theta, "theta", torch.float32, (w, 1 << k))
    _need(dtheta, "dtheta", torch.float32, (w, 1 << k))
    n_up = 0
    if dY is not None:
        if w % dy_group != 0:
            raise ValueError("dy_group must divide w")
        _need(dY, "dY", torch.float32, (w // dy_group, B))
    if up_terms is not None:
        n_up = up_terms.shape[0]
        _need(up_terms, "up_terms", torch.float32, (n_up, B))
        _need(up_off, "up_off", torch.int32, (w + 1,))
        if up_edge is not None:
            _need(up_edge, "up_edge", torch.int32, (n_up,))
    if dY_out is not None:
        _need(dY_out, "dY_out", torch.float32, (w, B))
    if order is not None:
        _need(order, "order", torch.int32, (w,))
    _check("bitlogic_lut_backward_bitrows", load().bitlogic_lut_backward_bitrows(
        _ptr(X), w_in, B, _ptr(conn), _ptr(theta), w, k, _node_code(node), _ptr(dY), int(dy_group),
        _ptr(up_terms), _ptr(up_off), _ptr(up_edge), n_up, _ptr(order), _ptr(dtheta), _ptr(dY_out),
        _stream(stream)))


def bitlogic_head_loss_ex(Y: torch.Tensor, labels: torch.Tensor, C: int, tau: float,
                          loss: torch.Tensor, workspace: torch.Tensor,
                          logits: Optional[torch.Tensor] = None,
                          dY: Optional[torch.Tensor] = None,
                          dY_grouped: Optional[torch.Tensor] = None, stream=None):
    w, B = Y.shape
    _need(Y, "Y", torch.float32, (w, B))
    _need(labels, "labels", torch.int32, (B,))
    _need(loss, "loss", torch.float32, (1,))
    if logits is not None:
        _need(logits, "logits", torch.float32, (B, C))
    if dY is not None:
        _need(dY, "dY", torch.float32, (w, B))
    if dY_grouped is not None:
        _need(dY_grouped, "dY_grouped", torch.float32, (C, B))
    if workspace is None or not workspace.is_cuda or workspace.dtype != torch.uint8:
        raise ValueError("workspace: uint8 CUDA tensor required")
    _check("bitlogic_head_loss_ex", load().bitlogic_head_loss_ex(
        _ptr(Y), w, B, C, float(tau), _ptr(labels), _ptr(logits), _ptr(loss), _ptr(dY),
        _ptr(dY_grouped), _ptr(workspace), workspace.numel(), _stream(stream)))


def bitlogic_head_loss_workspace(B: int, C: int) -> int:
    return int(load().bitlogic_head_loss_workspace(B, C))


def bitlogic_head_loss(Y: torch.Tensor, labels: torch.Tensor, C: int, tau: float,
                       loss: torch.Tensor, workspace: torch.Tensor,
                       logits: Optional[torch.Tensor] = None,
                       dY: Optional[torch.Tensor] = None, stream=None):
    w, B = Y.shape
    _need(Y, "Y", torch.float32, (w, B))
    _need(labels, "labels", torch.int32, (B,))
    _need(loss, "loss", torch.float32, (1,))
    if logits is not None:
        _need(logits, "logits", torch.float32, (B, C))
    if dY is not None:
        _need(dY, "dY", torch.float32, (w, B))
    if workspace is None or not workspace.is_cuda or workspace.dtype != torch.uint8:
        raise ValueError("workspace: uint8 CUDA tensor required")
    _check("bitlogic_head_loss", load().bitlogic_head_loss(
        _ptr(Y), w, B, C, float(tau), _ptr(labels), _ptr(logits), _ptr(loss), _ptr(dY),
        _ptr(workspace), workspace.numel(), _stream(stream)))


def bitlogic_head_loss_noalloc(Y: torch.Tensor, labels: torch.Tensor, C: int, tau: float,
                               loss: torch.Tensor, logits: Optional[torch.Tensor] = None,
                               dY: Optional[torch.Tensor] = None, stream=None):
    """bitlogic_head_loss with the library's fixed scratch instead of a
    caller workspace (for callers that cannot allocate device memory)."""
    w, B = Y.shape
    _need(Y, "Y", torch.float32, (w, B))
    _need(labels, "labels", torch.int32, (B,))
    _need(loss, "loss", torch.float32, (1,))
    if logits is not None:
        _need(logits, "logits", torch.float32, (B, C))
    if dY is not None:
        _need(dY, "dY", torch.float32, (w, B))
    _check("bitlogic_head_loss_noalloc", load().bitlogic_head_loss_noalloc(
        _ptr(Y), w, B, C, float(tau), _ptr(labels), _ptr(logits), _ptr(loss), _ptr(dY),
        _stream(stream)))


def bitlogic_binarize_tables(theta: torch.Tensor, table: torch.Tensor, stream=None):
    w, K = theta.shape
    k = K.bit_length() - 1
    _need(theta, "theta", torch.float32, (w, K))
    _need(table, "table", torch.int64, (w,))
    _check("bitlogic_binarize_tables", load().bitlogic_binarize_tables(
        _ptr(theta), w, k, _ptr(table), _stream(stream)))


def bitlogic_pack_bits(x: torch.Tensor, thresholds, xp: torch.Tensor, stream=None):
    N, d = x.shape
    buf, b = _thr_buf(thresholds)
    _need(x, "x", torch.uint8, (N, d))
    _need(xp, "xp", torch.int32, (d * b, (N + 31) // 32))
    _check("bitlogic_pack_bits", load().bitlogic_pack_bits(
        _ptr(x), N, d, buf, b, _ptr(xp), _stream(stream)))


def bitlogic_hard_forward(xp: torch.Tensor, N: int, conn: torch.Tensor, table: torch.Tensor,
                          yp: Optional[torch.Tensor] = None, C: int = 0,
                          counts: Optional[torch.Tensor] = None,
                          pred: Optional[torch.Tensor] = None, stream=None):
    w_in, W = xp.shape
    w, k = conn.shape
    if W != (N + 31) // 32:
        raise ValueError("xp has the wrong number of words for N")
    _need(xp, "xp", torch.int32, (w_in, W))
    _need(conn, "conn", torch.int32, (w, k))
    _need(table, "table", torch.int64, (w,))
    if yp is not None:
        _need(yp, "yp", torch.int32, (w, W))
    if counts is not None:
        _need(counts, "counts", torch.int32, (N, C))
    if pred is not None:
        _need(pred, "pred", torch.int32, (N,))
    _check("bitlogic_hard_forward", load().bitlogic_hard_forward(
        _ptr(xp), w_in, N, _ptr(conn), _ptr(table), w, k, _ptr(yp), C, _ptr(counts),
        _ptr(pred), _stream(stream)))


def bitlogic_build_csr(conn: np.ndarray, w_in: int) -> Tuple[np.ndarray, np.ndarray]:
    """Host call: inverse connectivity of int32 conn [w, k] -> (off, edge)."""
    conn = np.ascontiguousarray(conn, dtype=np.int32)
    w, k = conn.shape
    off = np.zeros(w_in + 1, np.int32)
    edge = np.zeros(w * k, np.int32)
    _check("bitlogic_build_csr", load().bitlogic_build_csr(
        conn.ctypes.data_as(_P), w, k, w_in, off.ctypes.data_as(_P), edge.ctypes.data_as(_P)))
    return off, edge


def bitlogic_adamw_update(theta: torch.Tensor, m: torch.Tensor, v: torch.Tensor, grad: torch.Tensor,
                          step: int, lr: float = 0.01, betas=(0.9, 0.999), eps: float = 1e-8,
                          weight_decay: float = 0.0, stream=None):
    """One AdamW step in place on theta, m, v (same shape, fp32, device)."""
    shape = tuple(theta.shape)
    for t, name in ((theta, "theta"), (m, "m"), (v, "v"), (grad, "grad")):
        _need(t, name, torch.float32, shape)
    _check("bitlogic_adamw_update", load().bitlogic_adamw_update(
        _ptr(theta), _ptr(m), _ptr(v), _ptr(grad), theta.numel(), int(step), float(lr),
        float(betas[0]), float(betas[1]), float(eps), float(weight_decay), _stream(stream)))


def bitlogic_degree_order(csr_off: np.ndarray) -> np.ndarray:
    """Host call: the nodes by decreasing CSR degree (ties by index)."""
    off = np.ascontiguousarray(csr_off, dtype=np.int32)
    n = off.shape[0] - 1
    order = np.zeros(max(n, 0), np.int32)
    _check("bitlogic_degree_order", load().bitlogic_degree_order(
        off.ctypes.data_as(_P), n, order.ctypes.data_as(_P)))
    return order


def bitlogic_csr_positions(csr_edge: np.ndarray) -> np.ndarray:
    """Host call: pos[csr_edge[p]] = p (the CSR position of every edge)."""
    edge = np.ascontiguousarray(csr_edge, dtype=np.int32)
    pos = np.zeros(edge.shape[0], np.int32)
    _check("bitlogic_csr_positions", load().bitlogic_csr_positions(
        edge.ctypes.data_as(_P), edge.shape[0], pos.ctypes.data_as(_P)))
    return pos


def bitlogic_device_error(stream=None) -> int:
    """Synchronizes the stream; returns 0 or the device index-flag status."""
    return int(load().bitlogic_device_error(_stream(stream)))
