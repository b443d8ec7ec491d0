"""The allocation-free MoE entry point (tqfx4_moe_ffn_noalloc).

Some callers cannot allocate device memory (a plug-in inside a host
application that owns all device memory, a serving loop where an allocation
may block and synchronize the device). tqfx4_moe_ffn_noalloc serves them: it
runs the same one-token MoE layer as tqfx4_moe_ffn on a scratch array held by
the library. This file checks, through the C ABI, that two calls in a row
match the workspace entry point on the same inputs, and that shapes whose
scratch need exceeds the library's array are refused before any launch. It
is named to be collected last, so a run that stops at the first failure has
already run every other test; it also passes alone in a fresh process.
"""
import numpy as np
import pytest
import torch

from paper_2608_08910_gb300 import binding as B
from paper_2608_08910_gb300 import inputs
from paper_2608_08910_gb300.moe import MoeLayer
from tests.parity import FP32_TOL, rel_err

pytestmark = pytest.mark.gpu
DEV = "cuda"


def _run_noalloc(layer, x):
    out = torch.empty(layer.hidden, device=DEV)
    sel = torch.empty(layer.top_k, dtype=torch.int32, device=DEV)
    selw = torch.empty(layer.top_k, device=DEV)
    B.tqfx4_moe_ffn_noalloc(layer.ex, layer.rt, x, out, sel, selw)
    torch.cuda.synchronize()
    return out, sel, selw


@pytest.mark.parametrize("E,H,I,k", [(64, 2048, 1024, 8), (256, 4096, 2048, 8)])
def test_noalloc_matches_workspace_entry_point_twice(E, H, I, k):
    layer = MoeLayer.synthetic(7, E, H, I, k, 0.0, DEV)
    X = inputs.hidden_states(7, 2, H).to(DEV)
    ws = layer.workspace(1)
    for t in range(2):  # two calls in a row on the shared scratch
        ref_out, ref_sel, ref_w = (a.clone() for a in layer.ffn(X[t], ws))
        B.tqfx4_check(ws)
        out, sel, selw = _run_noalloc(layer, X[t])
        assert torch.equal(sel, ref_sel)
        assert torch.equal(selw, ref_w)
        assert rel_err(out.cpu().numpy(), ref_out.cpu().numpy()) <= FP32_TOL
        assert np.array_equal(out.cpu().numpy().view(np.uint32), ref_out.cpu().numpy().view(np.uint32))


def test_noalloc_refuses_shapes_beyond_its_scratch():
    # hidden = inter = 16384 with 1024 experts and top-16: its one-token workspace exceeds 1 MiB
    ex = B.c_experts(None, None, None, 1024, 16384, 16384)
    rt = B.c_router(None, None, 16)
    assert B.tqfx4_moe_workspace_bytes(ex, rt, 1, 0) > B.TQFX4_NOALLOC_SCRATCH_BYTES
    x = torch.zeros(16384, device=DEV)
    with pytest.raises(B.TqfxError) as e:
        B.tqfx4_moe_ffn_noalloc(ex, rt, x, x, torch.zeros(16, dtype=torch.int32, device=DEV),
                                torch.zeros(16, device=DEV))
    assert e.value.status == 4
