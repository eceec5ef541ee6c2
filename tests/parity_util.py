"""Tolerances of the GPU-vs-oracle parity tests.

Integer, byte and bit outputs must match exactly.  fp32 forward outputs must
be within 1e-5 relative of the fp64 oracle; gradients within 1e-4 relative
plus 1e-6 absolute, element by element.  Because the gradients of these
workloads are themselves of order 1e-6..1e-3, gradients must in addition be
within 1e-4 of the tensor's largest oracle magnitude (a scale-aware bound
that the absolute term alone would not enforce).
"""
import numpy as np

FWD_RTOL = 1e-5
GRAD_RTOL = 1e-4
GRAD_ATOL = 1e-6


def as_np(t):
    if hasattr(t, "detach"):
        t = t.detach().cpu().numpy()
    return np.asarray(t)


def check_fwd(got, want, name="", atol=0.0):
    """1e-5 relative; ``atol`` adds an absolute term where the arithmetic
    gives no relative bound (hard table entries on fractional inputs, whose
    output can be an arbitrarily small corner weight)."""
    got = as_np(got).astype(np.float64)
    want = np.asarray(want, np.float64)
    assert got.shape == want.shape, (name, got.shape, want.shape)
    assert np.all(np.isfinite(got)), name
    err = np.abs(got - want)
    bad = err > FWD_RTOL * np.abs(want) + atol
    if bad.any():
        i = np.unravel_index(np.argmax(err - FWD_RTOL * np.abs(want)), want.shape)
        raise AssertionError(f"{name}: {bad.sum()} of {bad.size} outside 1e-5 rel + {atol} abs; worst at {i}: "
                             f"got {got[i]!r} want {want[i]!r}")
    return float((err / np.maximum(np.abs(want), 1e-300)).max()) if want.size else 0.0


def check_grad(got, want, name=""):
    got = as_np(got).astype(np.float64)
    want = np.asarray(want, np.float64)
    assert got.shape == want.shape, (name, got.shape, want.shape)
    assert np.all(np.isfinite(got)), name
    err = np.abs(got - want)
    bad = err > GRAD_ATOL + GRAD_RTOL * np.abs(want)
    if bad.any():
        i = np.unravel_index(np.argmax(err - GRAD_RTOL * np.abs(want)), want.shape)
        raise AssertionError(f"{name}: {bad.sum()} of {bad.size} outside 1e-4 rel + 1e-6 abs; "
                             f"worst at {i}: got {got[i]!r} want {want[i]!r}")
    scale = float(np.abs(want).max()) if want.size else 0.0
    if scale > 0:
        worst = float(err.max())
        assert worst <= GRAD_RTOL * scale, f"{name}: max error {worst} > 1e-4 * max|want| ({scale})"
        return worst / scale
    return 0.0


def check_exact(got, want, name=""):
    got = as_np(got)
    want = np.asarray(want)
    assert got.shape == want.shape, (name, got.shape, want.shape)
    if not np.array_equal(got, want):
        idx = np.argwhere(got != want)
        raise AssertionError(f"{name}: {len(idx)} mismatches, first at {idx[0].tolist()}")
