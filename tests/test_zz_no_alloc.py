"""The no-allocation W8A8 linear (w8a8_linear_noalloc) against the workspace one (w8a8_linear).

Callers that cannot allocate device memory use w8a8_linear_noalloc, which runs on a scratch array
built into the library.  These checks call it through the C ABI, twice in a row with different
inputs (the array keeps the previous call's contents, so the second call must not see them),
and require the same bits as w8a8_linear, the W8A8 tests' tolerance.  This file is collected last
so that a run stopping at the first failure has run every other test already; it also passes on
its own in a fresh process.
"""
import ctypes

import numpy as np
import pytest
import torch

import synth

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def B():
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    from paper_2608_28003_gb300 import build
    build.build()
    from paper_2608_28003_gb300 import binding
    return binding


def _call_noalloc(B, q, x):
    """One call through the C ABI (no workspace argument exists)."""
    M = x.shape[0]
    y = torch.empty(M, q.n, dtype=torch.bfloat16, device=x.device)
    wc = q.c()
    status = B.lib().w8a8_linear_noalloc(ctypes.byref(wc), ctypes.c_void_p(x.data_ptr()), M, None,
                                         ctypes.c_void_p(y.data_ptr()),
                                         ctypes.c_void_p(torch.cuda.current_stream().cuda_stream))
    assert status == 0, B.lib().w8a8_last_error()
    # no bounded wait gave up during the call
    status = B.lib().w8a8_linear_noalloc_check(ctypes.c_void_p(torch.cuda.current_stream().cuda_stream))
    assert status == 0, B.lib().w8a8_last_error()
    return y


@pytest.mark.parametrize("M,N,K", [(16, 6912, 1152), (1, 1152, 6912), (9, 1000, 1040)])
def test_noalloc_matches_workspace_linear_twice(B, M, N, K):
    x1_32, x1, ch = synth.activations(M, K, 8, seed=M + 1)
    x2_32, x2, _ = synth.activations(M, K, 8, seed=M + 2, channels=ch)
    _, w = synth.weight(N, K, seed=N)
    q = B.prepare_weights(w.cuda(), B.act_absmax(torch.cat([x1, x2]).cuda()))
    ref1 = B.linear(q, x1.cuda())
    ref2 = B.linear(q, x2.cuda())
    y1 = _call_noalloc(B, q, x1.cuda())
    y2 = _call_noalloc(B, q, x2.cuda())
    torch.cuda.synchronize()
    assert torch.equal(y1.view(torch.int16), ref1.view(torch.int16))
    assert torch.equal(y2.view(torch.int16), ref2.view(torch.int16))
    assert not torch.equal(y1, y2)


def test_noalloc_rejects_sizes_beyond_its_scratch(B):
    cap = B.lib().w8a8_linear_noalloc_capacity()
    assert cap == 8 << 20
    _, w = synth.weight(6912, 1152, seed=1)
    q = B.prepare_weights(w.cuda(), None, 0.5, False)
    x = torch.zeros(512, 1152, dtype=torch.bfloat16, device="cuda")
    y = torch.empty(512, 6912, dtype=torch.bfloat16, device="cuda")
    wc = q.c()
    status = B.lib().w8a8_linear_noalloc(ctypes.byref(wc), ctypes.c_void_p(x.data_ptr()), 512, None,
                                         ctypes.c_void_p(y.data_ptr()), None)
    assert status == 2 and b"scratch" in B.lib().w8a8_last_error()
