"""The allocation-free head entry point, bitlogic_head_loss_noalloc.

Some callers cannot allocate device memory (code hosted in another runtime
that owns the allocator, or loops with a fixed memory budget in which
cudaMalloc / cudaFree are not allowed).  For them the library keeps the
head's workspace in a fixed device array of its own.  These tests call that
entry point through the C ABI and check it against bitlogic_head_loss with a
caller workspace, on two different calls in a row (the shared array keeps
the previous call's contents).  This file is collected last on purpose.
"""
import ctypes

import numpy as np
import pytest
import torch

import paper_2602_07400_gb300 as bl
from parity_util import check_exact, check_fwd, check_grad

P = ctypes.c_void_p


def _ptr(t):
    return None if t is None else P(t.data_ptr())


def test_noalloc_rejects_sizes_beyond_its_scratch():
    # checked on the host before any CUDA call: no GPU needed
    lib = bl.load()
    fake = P(16)
    assert lib.bitlogic_head_loss_noalloc(fake, 8192 * 1000, 8192, 1000, 1.0, fake, None, fake,
                                          None, None) == -10
    assert "scratch" in bl.bitlogic_status_string(-10)
    assert lib.bitlogic_head_loss_noalloc(fake, 10, 0, 10, 1.0, fake, None, fake, None, None) == -2


def _case(C, g, B, tau, seed):
    rng = np.random.default_rng(seed)
    Y = torch.from_numpy(rng.random((C * g, B)).astype(np.float32)).cuda()
    labels = torch.from_numpy(rng.integers(0, C, size=B).astype(np.int32)).cuda()
    return Y, labels


def _reference(Y, labels, C, tau):
    w, B = Y.shape
    ws = torch.empty(bl.bitlogic_head_loss_workspace(B, C), dtype=torch.uint8, device="cuda")
    loss = torch.zeros(1, device="cuda")
    logits = torch.empty(B, C, device="cuda")
    dY = torch.empty(w, B, device="cuda")
    bl.bitlogic_head_loss(Y, labels, C, tau, loss, ws, logits=logits, dY=dY)
    return loss, logits, dY


@pytest.mark.gpu
def test_noalloc_head_matches_workspace_head_twice():
    lib = bl.load()
    stream = P(torch.cuda.current_stream().cuda_stream)
    # two different calls in a row: the second must not see the first's data
    for (C, g, B, tau, seed) in [(10, 80, 259, 20.0, 1), (100, 13, 1024, 100.0, 2)]:
        Y, labels = _case(C, g, B, tau, seed)
        w = C * g
        loss = torch.full((1,), np.nan, device="cuda")
        logits = torch.full((B, C), np.nan, device="cuda")
        dY = torch.full((w, B), np.nan, device="cuda")
        st = lib.bitlogic_head_loss_noalloc(_ptr(Y), w, B, C, tau, _ptr(labels), _ptr(logits),
                                            _ptr(loss), _ptr(dY), stream)
        assert st == 0, bl.bitlogic_status_string(st)
        ref_loss, ref_logits, ref_dY = _reference(Y, labels, C, tau)
        torch.cuda.synchronize()
        check_fwd(loss, ref_loss.cpu().numpy().astype(np.float64), "loss")
        check_fwd(logits, ref_logits.cpu().numpy().astype(np.float64), "logits")
        check_grad(dY, ref_dY.cpu().numpy().astype(np.float64), "dY")
        # without a logits buffer the logits go to the fixed scratch as well
        loss2 = torch.zeros(1, device="cuda")
        st = lib.bitlogic_head_loss_noalloc(_ptr(Y), w, B, C, tau, _ptr(labels), None,
                                            _ptr(loss2), None, stream)
        assert st == 0
        torch.cuda.synchronize()
        check_exact(loss2.cpu().numpy(), loss.cpu().numpy(), "loss without optional outputs")
    assert bl.bitlogic_device_error() == 0
