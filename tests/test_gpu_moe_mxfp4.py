"""GPU parity of tqfx4_moe_ffn_mxfp4 (one token through a routed-expert MoE
layer whose experts are MXFP4 blocks, Sec. 2.3) against the CPU oracle's
MoE with the MXFP4 dot pass: the selection exact, the routing weights and
the output bit-exact (the same binary32 schedules on both sides) and within
1e-4 relative."""
import numpy as np
import pytest
import torch

import oracle
from paper_2608_08910_gb300 import binding as B
from paper_2608_08910_gb300 import inputs
from paper_2608_08910_gb300.moe import MoeLayer
from tests.parity import FP32_TOL, rel_err

pytestmark = pytest.mark.gpu
DEV = "cuda"


def _oracle_experts(L, idx):
    ex = {}
    for e in np.unique(idx):
        ex[int(e)] = tuple(b.cpu().numpy() for b in L.expert_blocks(int(e)))
    return ex


@pytest.mark.parametrize("E,H,I,k,zipf", [(16, 512, 512, 4, 0.0), (32, 1024, 1536, 6, 1.1),
                                          (64, 2048, 1024, 8, 0.0)])
def test_moe_mxfp4_matches_oracle(E, H, I, k, zipf):
    L = MoeLayer.synthetic_mxfp4(E + H, E, H, I, k, zipf, DEV)
    ws = L.workspace(1)
    X = inputs.hidden_states(E + I, 3, H, DEV)
    Wr = L.router_w.cpu().numpy()
    bias = None if L.router_b is None else L.router_b.cpu().numpy()
    for t in range(X.shape[0]):
        out, sel, w = L.ffn(X[t], ws)
        B.tqfx4_check(ws)
        _, ridx, _ = oracle.router(Wr, bias, X[t].cpu().numpy(), k)
        ref, r_idx, r_w = oracle.moe_tokens(_oracle_experts(L, ridx), E, H, I, Wr, bias, k,
                                            X[t].cpu().numpy(), fmt="mxfp4")
        assert np.array_equal(sel.cpu().numpy(), r_idx[0])
        assert np.array_equal(w.cpu().numpy().view(np.uint32), r_w[0].view(np.uint32))
        got = out.cpu().numpy()
        assert np.array_equal(got.view(np.uint32), ref[0].view(np.uint32))
        assert rel_err(got, ref[0]) <= FP32_TOL


def test_moe_mxfp4_full_size_layer_sampled():
    # the 256-expert, hidden 4096, inter 2048, top-8 layer: two tokens
    E, H, I, k = 256, 4096, 2048, 8
    L = MoeLayer.synthetic_mxfp4(0, E, H, I, k, 0.0, DEV)
    ws = L.workspace(1)
    X = inputs.hidden_states(3, 2, H, DEV)
    Wr = L.router_w.cpu().numpy()
    for t in range(2):
        out, sel, w = L.ffn(X[t], ws)
        B.tqfx4_check(ws)
        ref, r_idx, _ = oracle.moe_tokens(_oracle_experts(L, sel.cpu().numpy()), E, H, I, Wr, None, k,
                                          X[t].cpu().numpy(), fmt="mxfp4")
        assert np.array_equal(sel.cpu().numpy(), r_idx[0])
        assert np.array_equal(out.cpu().numpy().view(np.uint32), ref[0].view(np.uint32))


def test_moe_mxfp4_argument_errors():
    L = MoeLayer.synthetic_mxfp4(1, 8, 512, 512, 2, 0.0, DEV)
    ws = L.workspace(1)
    x = inputs.hidden_states(2, 1, 512, DEV)[0]
    out = torch.empty(512, device=DEV)
    sel = torch.empty(2, dtype=torch.int32, device=DEV)
    w = torch.empty(2, device=DEV)
    with pytest.raises(B.TqfxError) as e:
        B.tqfx4_moe_ffn_mxfp4(L.ex, L.rt, None, out, sel, w, ws)
    assert e.value.status == 1
    bad = MoeLayer(L.gate, L.up, L.down, L.router_w, None, 8, 768, 512, 2, fmt="mxfp4")
    with pytest.raises(B.TqfxError) as e:  # hidden not a multiple of 512
        B.tqfx4_moe_ffn_mxfp4(bad.ex, bad.rt, x, out, sel, w, ws)
    assert e.value.status == 2
    with pytest.raises(B.TqfxError) as e:  # workspace too small
        B.tqfx4_moe_ffn_mxfp4(L.ex, L.rt, x, out, sel, w, ws[:64])
    assert e.value.status == 4
