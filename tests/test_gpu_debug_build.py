"""The format check and the debug build (TQFX4_DEBUG).

tqfx4_validate_blocks checks a tq2_0_fx4 matrix against the format: code
nibbles 0..8 and finite f16 row scales; a planted violation (a nibble of 15,
an infinite scale) must show as TQFX4_EDATA naming its block, with no fault.
The debug library validates every matrix an entry point reads and checks the
kernels' data-dependent indices; on valid inputs it must give the release
library's results bit for bit, and on a corrupted matrix it must report
TQFX4_EDATA from the validation (the dot pass itself never faults on a bad
nibble: it only computes a wrong sum).
"""
import ctypes as C

import numpy as np
import pytest
import torch

from paper_2608_08910_gb300 import binding as B
from paper_2608_08910_gb300 import build as libbuild
from paper_2608_08910_gb300 import inputs, ops
from paper_2608_08910_gb300.moe import MoeLayer

pytestmark = pytest.mark.gpu
DEV = "cuda"
K_VALIDATE = 14  # the kernel id the status word records for the format check
EDATA = 7


@pytest.fixture(scope="module")
def dbg():
    libbuild.build(debug=True)
    return B.load(B.DEBUG_LIB_PATH)


def status(ws):
    return ws[:12].view(torch.int32).cpu().tolist()


def packed(n, k, seed):
    ws = ops.workspace(B.TQFX4_STATUS_BYTES, DEV)
    return ops.pack_rtn(inputs.gemv_matrix(seed, n, k).to(DEV), ws)


def test_validate_accepts_packed_matrices():
    ws = ops.workspace(B.TQFX4_STATUS_BYTES, DEV)
    for n, k, seed in [(4, 256, 1), (1024, 1024, 2), (36, 768, 3)]:
        B.tqfx4_validate_blocks(packed(n, k, seed), n, k, ws)
    B.tqfx4_check(ws)


@pytest.mark.parametrize("where", ["nibble", "scale"])
def test_validate_reports_a_planted_violation(where):
    n, k = 64, 1024
    blocks = packed(n, k, 4)
    blk = 37  # block (row group 37 // 4, block 37 % 4) of the 16 x 4
    base = blk * B.TQFX4_BLOCK_BYTES
    if where == "nibble":
        blocks[base + 8 + 200] = (blocks[base + 8 + 200] & 0x0F) | 0xF0  # high nibble 15
    else:
        blocks[base + 2] = 0x00  # row scale 1 := +infinity (f16 0x7C00)
        blocks[base + 3] = 0x7C
    ws = ops.workspace(B.TQFX4_STATUS_BYTES, DEV)
    B.tqfx4_validate_blocks(blocks, n, k, ws)
    torch.cuda.synchronize()
    st = status(ws)
    assert st == [EDATA, K_VALIDATE, blk], st
    with pytest.raises(B.TqfxError) as e:
        B.tqfx4_check(ws)
    assert e.value.status == EDATA


def _gemv(L, blocks, n, k, x, ws):
    y = torch.empty(n, device=DEV)
    rc = L.tqfx4_gemv_x(blocks.data_ptr(), n, k, x.data_ptr(), y.data_ptr(), None, None, None, ws.data_ptr(),
                        ws.numel(), torch.cuda.current_stream().cuda_stream)
    assert rc == 0
    return y


def test_debug_build_gives_the_release_bits(dbg):
    n, k = 512, 2048
    blocks = packed(n, k, 5)
    x = inputs.hidden_states(5, 1, k)[0].to(DEV)
    ws_r = ops.workspace(B.TQFX4_STATUS_BYTES, DEV)
    ws_d = ops.workspace(B.TQFX4_STATUS_BYTES, DEV)
    y_r = _gemv(B.lib(), blocks, n, k, x, ws_r)
    y_d = _gemv(dbg, blocks, n, k, x, ws_d)
    torch.cuda.synchronize()
    assert status(ws_d) == [0, 0, 0]
    assert torch.equal(y_r.view(torch.int32), y_d.view(torch.int32))
    # one token through a small MoE layer, decode and grouped
    layer = MoeLayer.synthetic(9, 16, 512, 512, 4, 0.0, DEV)
    xm = inputs.hidden_states(9, 6, 512).to(DEV)
    for grouped in (False, True):
        outs = []
        for L in (B.lib(), dbg):
            ws = layer.workspace(6 if grouped else 1)
            stream = torch.cuda.current_stream().cuda_stream
            if grouped:
                out = torch.empty(6, 512, device=DEV)
                sel = torch.empty(6, 4, dtype=torch.int32, device=DEV)
                w = torch.empty(6, 4, device=DEV)
                rc = L.tqfx4_moe_grouped(C.byref(layer.ex), C.byref(layer.rt), xm.data_ptr(), 6, out.data_ptr(),
                                         sel.data_ptr(), w.data_ptr(), B.TQFX4_PATH_PREFILL, ws.data_ptr(),
                                         ws.numel(), stream)
            else:
                out = torch.empty(512, device=DEV)
                sel = torch.empty(4, dtype=torch.int32, device=DEV)
                w = torch.empty(4, device=DEV)
                rc = L.tqfx4_moe_ffn(C.byref(layer.ex), C.byref(layer.rt), xm[0].data_ptr(), out.data_ptr(),
                                     sel.data_ptr(), w.data_ptr(), ws.data_ptr(), ws.numel(), stream)
            assert rc == 0
            torch.cuda.synchronize()
            assert status(ws) == [0, 0, 0], (grouped, status(ws))
            outs.append((out.clone(), sel.clone(), w.clone()))
        for a, b in zip(*outs):
            assert torch.equal(a.view(torch.int32), b.view(torch.int32)), grouped


def test_debug_build_reports_a_corrupted_matrix(dbg):
    n, k = 256, 1024
    blocks = packed(n, k, 6)
    blk = 100
    blocks[blk * B.TQFX4_BLOCK_BYTES + 8 + 3] = 0x9A  # nibbles 10 and 9
    x = inputs.hidden_states(6, 1, k)[0].to(DEV)
    ws = ops.workspace(B.TQFX4_STATUS_BYTES, DEV)
    _gemv(dbg, blocks, n, k, x, ws)
    torch.cuda.synchronize()
    assert status(ws) == [EDATA, K_VALIDATE, blk], status(ws)
    # the release library computes through it without a check (and without a fault)
    ws_r = ops.workspace(B.TQFX4_STATUS_BYTES, DEV)
    _gemv(B.lib(), blocks, n, k, x, ws_r)
    torch.cuda.synchronize()
    assert status(ws_r) == [0, 0, 0]
