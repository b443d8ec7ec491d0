"""GPU parity of the tied alternating solver (tqfx4_pack with
TQFX4_SRC_F32_TIED, Sec. 2.1) against the CPU oracle, through the C ABI: the
blocks (f16 scales and nibble codes) must be bit-exact, for weights whose
scales span many orders of magnitude (f16 subnormal to large scales), the
Student-t expert projections of the benchmark layers, ragged shapes, an
all-zero matrix and the iteration cap; non-finite weights are reported."""
import numpy as np
import pytest
import torch

import oracle
from paper_2608_08910_gb300 import binding as B
from paper_2608_08910_gb300 import inputs, ops

pytestmark = pytest.mark.gpu
DEV = "cuda"


@pytest.fixture(scope="module")
def ws():
    return ops.workspace(B.TQFX4_STATUS_BYTES)


@pytest.mark.parametrize("n,k", [(4, 256), (1024, 1024), (132, 768), (260, 1280), (8, 16384), (36, 256 * 33)])
def test_pack_tied_bit_exact(n, k, ws):
    w = inputs.log_uniform_scale_matrix(7 * n + k, n, k)
    ref, iters = oracle.pack_tied(w.numpy(), B.TQFX4_TIED_MAX_ITER, with_iters=True)
    got = ops.pack_tied(w.to(DEV), ws).cpu().numpy()
    B.tqfx4_check(ws)
    assert np.array_equal(got, ref)


def test_pack_tied_student_t_expert_bit_exact(ws):
    w = inputs.expert_matrix(0, 5, inputs.PROJ_DOWN, 4096, 2048)
    ref, iters = oracle.pack_tied(w.numpy(), B.TQFX4_TIED_MAX_ITER, with_iters=True)
    got = ops.pack_tied(w.to(DEV), ws).cpu().numpy()
    B.tqfx4_check(ws)
    assert np.array_equal(got, ref)
    assert (iters > 0).mean() > 0.5  # most blocks move off the round-to-nearest fit
    assert not np.array_equal(got, ops.pack_rtn(w.to(DEV), ws).cpu().numpy())


def test_pack_tied_zero_and_nonfinite(ws):
    w = torch.zeros(8, 512)
    got = ops.pack_tied(w.to(DEV), ws).cpu().numpy()
    B.tqfx4_check(ws)
    assert np.array_equal(got, oracle.pack_rtn(w.numpy()))
    w[2, 7] = float("inf")
    ops.pack_tied(w.to(DEV), ws)
    with pytest.raises(B.TqfxError) as e:
        B.tqfx4_check(ws)
    assert e.value.status == 7
    B.tqfx4_check(ws)  # cleared


def test_gemv_on_tied_blocks_matches_oracle(ws):
    # the dot pass is format-agnostic: tied blocks go through the same GEMV
    n, k = 2048, 4096
    w = inputs.expert_matrix(1, 2, inputs.PROJ_GATE, 4096, 2048)
    x = inputs.hidden_states(3, 1, k)[0]
    blocks = ops.pack_tied(w.to(DEV), ws)
    ref_blocks = oracle.pack_tied(w.numpy())
    assert np.array_equal(blocks.cpu().numpy(), ref_blocks)
    rq, rda, _ = oracle.quantize_act(x.numpy())
    ry, rS = oracle.gemv(ref_blocks, n, k, rq, rda)
    q, da, bs = ops.quantize_act(x.to(DEV), ws)
    y, S = ops.gemv(blocks, n, k, q, da, bs, ws, block_sums=True)
    B.tqfx4_check(ws)
    assert np.array_equal(S.cpu().numpy(), rS)
    assert np.array_equal(y.cpu().numpy().view(np.uint32), ry.view(np.uint32))
