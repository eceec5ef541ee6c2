"""The allocation-free head entry point, bitlogic_head_loss_noalloc.

Some callers cannot allocate device memory (code hosted in another runtime
that owns the allocator, or loops with a fixed memory budget in which
cudaMalloc / cudaFree are not allowed).  For them the library keeps the
head's workspace in a fixed 8 MiB device array of its own.  These tests call
that entry point through the C ABI and check it against
bitlogic_head_loss with a caller workspace and against the oracle, on calls
in a row (the shared array keeps the previous call's contents), including
the largest batch whose workspace fits the array and a shape that uses every
row-split slot of the workspace.  This file is collected last on purpose.
"""
import ctypes

import numpy as np
import pytest
import torch

import oracle
import paper_2602_07400_gb300 as bl
from parity_util import check_exact, check_fwd, check_grad

P = ctypes.c_void_p
SCRATCH_BYTES = 8 << 20


def _ptr(t):
    return None if t is None else P(t.data_ptr())


def _largest_batch(C):
    """Largest B whose head workspace fits the fixed scratch (host-only
    size query, bisection on the library's own size function)."""
    lo, hi = 1, 1 << 24
    while hi - lo > 1:
        mid = (lo + hi) // 2
        if bl.bitlogic_head_loss_workspace(mid, C) <= SCRATCH_BYTES:
            lo = mid
        else:
            hi = mid
    return lo


def test_noalloc_rejects_sizes_beyond_its_scratch():
    # checked on the host before any CUDA call: no GPU needed
    lib = bl.load()
    fake = P(16)
    assert lib.bitlogic_head_loss_noalloc(fake, 8192 * 1000, 8192, 1000, 1.0, fake, None, fake,
                                          None, None) == -10
    assert "scratch" in bl.bitlogic_status_string(-10)
    assert lib.bitlogic_head_loss_noalloc(fake, 10, 0, 10, 1.0, fake, None, fake, None, None) == -2


@pytest.mark.parametrize("C", [1, 10, 100, 1000])
def test_noalloc_size_limit_is_exact(C):
    # one sample past the largest batch that fits is refused with -10; the
    # refusal comes from the host-side size check, before any CUDA call
    lib = bl.load()
    fake = P(16)
    B = _largest_batch(C)
    assert bl.bitlogic_head_loss_workspace(B, C) <= SCRATCH_BYTES < bl.bitlogic_head_loss_workspace(B + 1, C)
    assert lib.bitlogic_head_loss_noalloc(fake, C, B + 1, C, 1.0, fake, None, fake, None, None) == -10


def _case(C, g, B, seed):
    rng = np.random.default_rng(seed)
    Y = torch.from_numpy(rng.random((C * g, B)).astype(np.float32)).cuda()
    labels = torch.from_numpy(rng.integers(0, C, size=B).astype(np.int32)).cuda()
    return Y, labels


def _workspace_head(Y, labels, C, tau):
    w, B = Y.shape
    ws = torch.empty(bl.bitlogic_head_loss_workspace(B, C), dtype=torch.uint8, device="cuda")
    loss = torch.zeros(1, device="cuda")
    logits = torch.empty(B, C, device="cuda")
    dY = torch.empty(w, B, device="cuda")
    bl.bitlogic_head_loss(Y, labels, C, tau, loss, ws, logits=logits, dY=dY)
    return loss, logits, dY


def _noalloc_matches(lib, stream, C, g, B, tau, seed):
    Y, labels = _case(C, g, B, seed)
    w = C * g
    loss = torch.full((1,), np.nan, device="cuda")
    logits = torch.full((B, C), np.nan, device="cuda")
    dY = torch.full((w, B), np.nan, device="cuda")
    st = lib.bitlogic_head_loss_noalloc(_ptr(Y), w, B, C, tau, _ptr(labels), _ptr(logits),
                                        _ptr(loss), _ptr(dY), stream)
    assert st == 0, bl.bitlogic_status_string(st)
    ref_loss, ref_logits, ref_dY = _workspace_head(Y, labels, C, tau)
    torch.cuda.synchronize()
    # the same kernels on the same inputs: bit for bit the workspace head
    check_exact(loss.cpu().numpy(), ref_loss.cpu().numpy(), "loss vs workspace head")
    check_exact(logits.cpu().numpy(), ref_logits.cpu().numpy(), "logits vs workspace head")
    check_exact(dY.cpu().numpy(), ref_dY.cpu().numpy(), "dY vs workspace head")
    # and within the parity tolerances of the oracle
    o_logits, o_loss, o_dY = oracle.head_loss(Y.cpu().numpy(), labels.cpu().numpy(), C, tau)
    check_fwd(loss, np.array([o_loss]), "loss vs oracle")
    check_fwd(logits, o_logits, "logits vs oracle")
    check_grad(dY, o_dY, "dY vs oracle")
    # without a logits buffer the logits go to the fixed scratch as well
    loss2 = torch.zeros(1, device="cuda")
    st = lib.bitlogic_head_loss_noalloc(_ptr(Y), w, B, C, tau, _ptr(labels), None,
                                        _ptr(loss2), None, stream)
    assert st == 0
    torch.cuda.synchronize()
    check_exact(loss2.cpu().numpy(), loss.cpu().numpy(), "loss without optional outputs")


@pytest.mark.gpu
def test_noalloc_head_matches_workspace_head_and_oracle_twice():
    lib = bl.load()
    stream = P(torch.cuda.current_stream().cuda_stream)
    # two different calls in a row: the second must not see the first's data
    for (C, g, B, tau, seed) in [(10, 80, 259, 20.0, 1), (100, 13, 1024, 100.0, 2)]:
        _noalloc_matches(lib, stream, C, g, B, tau, seed)
    assert bl.bitlogic_device_error() == 0


@pytest.mark.gpu
def test_noalloc_head_at_its_size_limits():
    lib = bl.load()
    stream = P(torch.cuda.current_stream().cuda_stream)
    # row splits of the group sum: 10 classes of 2048 rows over 1024 samples
    # (split while the grid fits one wave), and over 256 samples (four
    # splits: every split slot of the workspace is written and read)
    _noalloc_matches(lib, stream, 10, 2048, 1024, 50.0, 3)
    _noalloc_matches(lib, stream, 10, 2048, 256, 50.0, 6)
    # the largest batch of 10 classes whose workspace fits the 8 MiB array,
    # rounded down to a multiple of 4 (the vector group sum)
    B = _largest_batch(10) // 4 * 4
    _noalloc_matches(lib, stream, 10, 3, B, 10.0, 4)
    # and a ragged batch right at the limit (scalar group sum)
    B = _largest_batch(7)
    if B % 4 == 0:
        B -= 1
    _noalloc_matches(lib, stream, 7, 2, B, 3.0, 5)
    assert bl.bitlogic_device_error() == 0
