"""Failure detection on the GPU without a fault.

Every wait in the library's kernels is bounded: a copy that never arrives,
or a peer that never signals, makes the waiting warp record TQFX4_ETIMEOUT
in the workspace's status word and return, instead of hanging the GPU.
tqfx4_selftest_wait_timeout runs the streaming engine's consume loop on a
ring whose copies were never issued, with a short budget (10^6 cycles), so
that this path runs for real: the status must come back as ETIMEOUT from
tqfx4_check, the word must be cleared by that check, and the next ordinary
call on the same context and workspace must succeed and be correct.
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2608_08910_gb300 import binding as B
from paper_2608_08910_gb300 import inputs, ops

pytestmark = pytest.mark.gpu
DEV = "cuda"


def test_bounded_wait_reports_timeout_and_the_context_stays_usable():
    ws = ops.workspace(B.TQFX4_STATUS_BYTES)
    B.tqfx4_selftest_wait_timeout(ws)
    with pytest.raises(B.TqfxError) as e:
        B.tqfx4_check(ws)
    assert e.value.status == 6  # TQFX4_ETIMEOUT
    assert "selftest" in str(e.value)
    B.tqfx4_check(ws)  # the check cleared the word
    # an ordinary GEMV afterwards, on the same workspace: correct bit for bit
    n, k = 64, 1024
    w = inputs.gemv_matrix(9, n, k)
    x = inputs.hidden_states(9, 1, k)[0]
    blocks = ops.pack_rtn(w.to(DEV), ws)
    q, da, bs = ops.quantize_act(x.to(DEV), ws)
    y = ops.gemv(blocks, n, k, q, da, bs, ws)
    B.tqfx4_check(ws)
    rq, rda, _ = oracle.quantize_act(x.numpy())
    ry, _ = oracle.gemv(oracle.pack_rtn(w.numpy()), n, k, rq, rda)
    assert np.array_equal(y.cpu().numpy().view(np.uint32), ry.view(np.uint32))


def test_timeout_twice_in_a_row():
    ws = ops.workspace(B.TQFX4_STATUS_BYTES)
    for _ in range(2):
        B.tqfx4_selftest_wait_timeout(ws)
        with pytest.raises(B.TqfxError) as e:
            B.tqfx4_check(ws)
        assert e.value.status == 6
    torch.cuda.synchronize()
