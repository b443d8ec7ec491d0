"""GPU tests of the expert tier (experts in pinned host memory, device slots
filled on a miss) and of the two-call decode it uses (tqfx4_moe_route, then
tqfx4_moe_experts over caller-given block pointers).

The paper's streamed store serves an expert from wherever it is cached with
the same bytes and the same kernels, so outputs do not depend on residency
(Sec. 2.2, property iii). Here that is checked bit for bit: the tier's
outputs, selections and weights equal the resident tqfx4_moe_ffn's for every
token, also when the slab holds only top_k experts and evicts.
The two-call decode and the tier are also checked against the CPU oracle
directly: their outputs within 1e-4 relative of the oracle's MoE (and bit for
bit, since the float schedules are the same), on the small layer and on the
256-expert benchmark layer.
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2608_08910_gb300 import binding as B
from paper_2608_08910_gb300 import inputs
from paper_2608_08910_gb300.moe import MoeLayer
from paper_2608_08910_gb300.tier import ExpertTier
from tests.parity import FP32_TOL, oracle_experts, rel_err

pytestmark = pytest.mark.gpu
DEV = "cuda"


def _bits(t):
    return t.cpu().numpy().view(np.uint32)


def _oracle_out(L, seed, x, sel):
    """The oracle's MoE output for token x, if its own routing equals `sel`
    (else None: a near-tie, accepted by the selection tests)."""
    Wr = L.router_w.cpu().numpy()
    bias = None if L.router_b is None else L.router_b.cpu().numpy()
    xn = x.cpu().numpy()
    _, ridx, _ = oracle.router(Wr, bias, xn, L.top_k)
    if not np.array_equal(ridx, sel):
        return None
    ex = oracle_experts(seed, ridx, L.hidden, L.inter)
    ref, _, _ = oracle.moe_tokens(ex, L.n_experts, L.hidden, L.inter, Wr, bias, L.top_k, xn)
    return ref[0]


@pytest.fixture(scope="module")
def small():
    return MoeLayer.synthetic(41, 32, 1024, 512, 6, 1.1, DEV)


def test_route_then_experts_equals_ffn(small):
    L = small
    ws = L.workspace(1)
    X = inputs.hidden_states(41, 4, L.hidden, DEV)
    K = L.top_k
    for t in range(X.shape[0]):
        ref_out, ref_sel, ref_w = [v.clone() for v in L.ffn(X[t], ws)]
        sel = torch.empty(K, dtype=torch.int32, device=DEV)
        w = torch.empty(K, device=DEV)
        B.tqfx4_moe_route(L.ex, L.rt, X[t], sel, w, ws)
        assert torch.equal(sel, ref_sel) and np.array_equal(_bits(w), _bits(ref_w))
        # pointers into the stacked layout: exactly what tqfx4_moe_ffn reads
        ptrs = torch.tensor([int(buf.data_ptr()) + int(e) * mb
                             for buf, mb in ((L.gate, L.mb_gu), (L.up, L.mb_gu), (L.down, L.mb_d))
                             for e in sel.tolist()], dtype=torch.int64, device=DEV)
        out = torch.empty(L.hidden, device=DEV)
        B.tqfx4_moe_experts(L.ex, L.rt, ptrs, out, ws)
        B.tqfx4_check(ws)
        assert np.array_equal(_bits(out), _bits(ref_out))
        if t < 2:  # against the oracle itself
            ref = _oracle_out(L, 41, X[t], sel.cpu().numpy())
            if ref is not None:
                assert rel_err(out.cpu().numpy(), ref) <= FP32_TOL
                assert np.array_equal(_bits(out), ref.view(np.uint32))


@pytest.mark.parametrize("slots", [6, 12])
def test_tier_outputs_equal_resident(small, slots):
    L = small
    ws = L.workspace(1)
    tier = ExpertTier(L, slots)
    X = inputs.hidden_states(43, 12, L.hidden, DEV)
    K = L.top_k
    for t in range(X.shape[0]):
        ref_out, ref_sel, ref_w = [v.clone() for v in L.ffn(X[t], ws)]
        out = torch.empty(L.hidden, device=DEV)
        sel = torch.empty(K, dtype=torch.int32, device=DEV)
        w = torch.empty(K, device=DEV)
        tier.ffn(X[t], ws, out, sel, w)
        B.tqfx4_check(ws)
        assert torch.equal(sel, ref_sel)
        assert np.array_equal(_bits(w), _bits(ref_w))
        assert np.array_equal(_bits(out), _bits(ref_out))
    assert tier.lookups == 12 * K
    assert slots < tier.misses < tier.lookups  # slots were evicted and refilled, and some lookups hit


def test_tier_full_size_layer():
    # the 256-expert benchmark layer: two tokens through a top_k-slot slab
    L = MoeLayer.synthetic(0, 256, 4096, 2048, 8, 0.0, DEV)
    ws = L.workspace(1)
    tier = ExpertTier(L, 8)
    X = inputs.hidden_states(7, 2, 4096, DEV)
    compared = 0
    for t in range(2):
        ref_out = L.ffn(X[t], ws)[0].clone()
        out = torch.empty(4096, device=DEV)
        sel = torch.empty(8, dtype=torch.int32, device=DEV)
        tier.ffn(X[t], ws, out, sel, torch.empty(8, device=DEV))
        B.tqfx4_check(ws)
        assert np.array_equal(_bits(out), _bits(ref_out))
        ref = _oracle_out(L, 0, X[t], sel.cpu().numpy())  # the tier against the oracle
        if ref is not None:
            assert rel_err(out.cpu().numpy(), ref) <= FP32_TOL
            assert np.array_equal(_bits(out), ref.view(np.uint32))
            compared += 1
    assert compared >= 1


def test_experts_argument_errors(small):
    L = small
    ws = L.workspace(1)
    out = torch.empty(L.hidden, device=DEV)
    with pytest.raises(B.TqfxError) as e:
        B.tqfx4_moe_experts(L.ex, L.rt, None, out, ws)
    assert e.value.status == 1
    with pytest.raises(B.TqfxError) as e:
        B.tqfx4_moe_experts(L.ex, L.rt, torch.zeros(64, dtype=torch.uint8, device=DEV)[1:], out, ws)
    assert e.value.status == 3
    with pytest.raises(B.TqfxError) as e:
        B.tqfx4_moe_route(L.ex, L.rt, None, None, None, ws)
    assert e.value.status == 1
