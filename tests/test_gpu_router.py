"""GPU parity of the screened router that large batches use (an fp32 GEMM with
a rigorous error bound, then compensated logits for the experts that can
still reach a token's top k): its selection and weights must equal those of
the exact per-token router, bit for bit, also where logits tie exactly, and
every logit it leaves approximate must lie within its bound of the oracle's.
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2608_08910_gb300 import binding as B
from paper_2608_08910_gb300 import inputs
from paper_2608_08910_gb300.moe import MoeLayer
from tests.parity import check_selection, selection_tolerance

pytestmark = pytest.mark.gpu
DEV = "cuda"
SCREEN_T = 300  # batches of at least 256 tokens are screened


def grouped_and_exact(layer, X, sample):
    T = X.shape[0]
    ws = layer.workspace(T)
    OUT, sel, selw = layer.grouped(X.to(DEV), ws, B.TQFX4_PATH_PREFILL)
    B.tqfx4_check(ws)
    wsd = layer.workspace(1)
    for t in sample:
        _, s, w = layer.ffn(X[t].to(DEV), wsd)
        assert np.array_equal(s.cpu().numpy(), sel[t].cpu().numpy()), t
        assert np.array_equal(w.cpu().numpy().view(np.uint32), selw[t].cpu().numpy().view(np.uint32)), t
    return ws, sel.cpu().numpy()


def test_screened_selection_equals_exact_router():
    layer = MoeLayer.synthetic(21, 64, 1024, 512, 8, 0.5, DEV)
    X = inputs.hidden_states(21, SCREEN_T, 1024)
    grouped_and_exact(layer, X, sample=range(0, SCREEN_T, 7))


def test_screened_router_exact_ties():
    # experts 2j and 2j+1 share a router row: every logit ties with its twin,
    # and the lower index must win wherever the pair straddles the top-k edge
    layer = MoeLayer.synthetic(22, 32, 512, 512, 5, 0.0, DEV)
    w = layer.router_w.view(32, 512)
    w[1::2] = w[0::2]
    X = inputs.hidden_states(22, SCREEN_T, 512)
    ws, sel = grouped_and_exact(layer, X, sample=range(0, SCREEN_T, 5))
    Wr = layer.router_w.cpu().numpy()
    for t in range(0, SCREEN_T, 13):
        logits, idx, _ = oracle.router(Wr, None, X[t].numpy(), 5)
        assert np.array_equal(np.sort(sel[t]), np.sort(idx)), t


def test_screened_logits_within_bound():
    E, H, k = 128, 2048, 8
    layer = MoeLayer.synthetic(23, E, H, 512, k, 1.1, DEV)
    X = inputs.hidden_states(23, SCREEN_T, H)
    ws = layer.workspace(SCREEN_T)
    OUT, sel, selw = layer.grouped(X.to(DEV), ws, B.TQFX4_PATH_PREFILL)
    B.tqfx4_check(ws)
    hi = layer.view(ws, "logits", torch.float32, (SCREEN_T, E), tokens=SCREEN_T, grouped=1).cpu().numpy()
    lo = layer.view(ws, "logits_lo", torch.float32, (SCREEN_T, E), tokens=SCREEN_T, grouped=1).cpu().numpy()
    Wr = layer.router_w.cpu().numpy().astype(np.float64)
    bias = layer.router_b.cpu().numpy()
    Xn = X.numpy().astype(np.float64)
    gamma = H * 2.0 ** -24 / (1 - H * 2.0 ** -24)
    nw = np.linalg.norm(Wr, axis=1)
    sel = sel.cpu().numpy()
    for t in range(0, SCREEN_T, 11):
        logits, _, _ = oracle.router(Wr.astype(np.float32), bias, X[t].numpy(), k)
        got = hi[t].astype(np.float64) + lo[t]
        bound = gamma * np.linalg.norm(Xn[t]) * nw + 2.0 ** -22 * np.abs(logits)
        assert np.all(np.abs(got - logits) <= bound), t
        # the selected experts carry compensated logits
        tol = selection_tolerance(Wr.astype(np.float32), X[t].numpy(), bias)
        assert np.all(np.abs(got[sel[t]] - logits[sel[t]]) <= tol[sel[t]])
        check_selection(sel[t], logits, tol, k)
