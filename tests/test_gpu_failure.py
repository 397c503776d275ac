"""Failure detection without a GPU fault: the device error word of a workspace.

Every bounded device-side wait that gives up sets a bit of the workspace's error word (at a fixed
offset in its reserved region) and returns; w8a8_workspace_check reads and clears it.  Here the bit
is written from the host, as a kernel's timeout would leave it, so no wait is made to run out on
the GPU: the check must report W8A8_ERR_TIMEOUT once, clear the word, and the workspace must then
serve a linear whose output is unchanged.
"""
import ctypes

import numpy as np
import pytest
import torch

import synth

pytestmark = pytest.mark.gpu

ERR_WORD_OFFSET = 36864  # byte offset of the error word inside the reserved region


@pytest.fixture(scope="module")
def B():
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    from paper_2608_28003_gb300 import build
    build.build()
    from paper_2608_28003_gb300 import binding
    return binding


def _check(B, ws):
    return B.lib().w8a8_workspace_check(ctypes.c_void_p(ws.data_ptr()),
                                        ctypes.c_void_p(torch.cuda.current_stream().cuda_stream))


@pytest.mark.parametrize("bits", [1, 2, 4, 7])
def test_error_word_reported_once_then_cleared(B, bits):
    ws = torch.zeros(B.WS_RESERVED, dtype=torch.uint8, device="cuda")
    assert _check(B, ws) == 0
    ws[ERR_WORD_OFFSET:ERR_WORD_OFFSET + 4] = torch.tensor(np.array([bits], np.uint32).view(np.uint8))
    assert _check(B, ws) == 6  # W8A8_ERR_TIMEOUT
    assert b"gave up" in B.lib().w8a8_last_error()
    assert int(ws[ERR_WORD_OFFSET:ERR_WORD_OFFSET + 4].view(torch.int32).item()) == 0
    assert _check(B, ws) == 0


def test_workspace_usable_after_a_reported_timeout(B):
    """A linear through a workspace whose error word was set and then checked gives the same bits
    as one through a fresh workspace."""
    x32, x, _ = synth.activations(16, 1152, 8, seed=3)
    _, w = synth.weight(6912, 1152, seed=3)
    q = B.prepare_weights(w.cuda(), B.act_absmax(x.cuda()))
    ref = B.linear(q, x.cuda(), ws=B.Workspace())
    ws = B.Workspace()
    ws.get(B._size("w8a8_linear_workspace_size", 16, 6912, 1152))  # sized before the bit is set
    ws.buf[ERR_WORD_OFFSET:ERR_WORD_OFFSET + 4] = torch.tensor(np.array([1], np.uint32).view(np.uint8))
    with pytest.raises(B.W8A8Error):
        B.workspace_check(ws)
    y = B.linear(q, x.cuda(), ws=ws)
    B.workspace_check(ws)
    assert torch.equal(y.view(torch.int16), ref.view(torch.int16))
