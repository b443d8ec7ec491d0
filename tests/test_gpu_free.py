"""GPU parity of the free-scale two-plane format (Table 1's free-scale K=2
row: two trit planes with two f16 scales, 4.125 bits/weight) against the CPU
oracle, through the C ABI: packed blocks, the int32 plane sums S1 and S2 and
the fp32 outputs bit-exact (the same binary32 schedule on both sides)."""
import numpy as np
import pytest
import torch

import oracle
from paper_2608_08910_gb300 import binding as B
from paper_2608_08910_gb300 import inputs, ops
from tests.parity import FP32_TOL, rel_err

pytestmark = pytest.mark.gpu
DEV = "cuda"

# a single block, expert shapes, odd block counts per row, k above 32 blocks
# (two pairs per lane and more), the largest k
SHAPES = [(4, 256), (64, 1024), (132, 768), (2048, 4096), (4096, 2048), (36, 256 * 33), (12, 256 * 7),
          (8, B.TQFX4_MAX_K)]


@pytest.fixture(scope="module")
def ws():
    return ops.workspace(B.TQFX4_STATUS_BYTES)


def _planes(seed, n, k, dev="cpu"):
    t1, t2, s1 = inputs.trit_planes(seed, n, k, dev)
    s2 = inputs.trit_planes(seed + 1, n, k, dev)[2]
    return t1, t2, s1.view(torch.int16), s2.view(torch.int16)


def _np16(t):
    return t.cpu().numpy().view(np.uint16)


@pytest.mark.parametrize("n,k", SHAPES)
def test_pack_and_gemv_bit_exact(n, k, ws):
    t1, t2, a1, a2 = _planes(n + k, n, k)
    ref = oracle.pack_free(t1.numpy(), t2.numpy(), _np16(a1), _np16(a2))
    blocks = ops.pack_free(t1.to(DEV), t2.to(DEV), a1.to(DEV), a2.to(DEV), ws)
    B.tqfx4_check(ws)
    assert np.array_equal(blocks.cpu().numpy(), ref)
    x = inputs.hidden_states(n + 2 * k, 1, k)[0]
    q, da, bs = oracle.quantize_act(x.numpy())
    ry, rS1, rS2 = oracle.free_gemv(ref, n, k, q, da)
    y, S1, S2 = ops.gemv_free(blocks, n, k, torch.from_numpy(q).to(DEV), torch.from_numpy(da).to(DEV),
                              torch.from_numpy(bs).to(DEV), ws, block_sums=True)
    B.tqfx4_check(ws)
    assert np.array_equal(S1.cpu().numpy(), rS1) and np.array_equal(S2.cpu().numpy(), rS2)
    got = y.cpu().numpy()
    assert np.array_equal(got.view(np.uint32), ry.view(np.uint32))
    assert rel_err(got, ry) <= FP32_TOL


def test_gemv_large_sampled(ws):
    # 131072 x 4096 (277 MB of blocks, larger than L2), device-quantized activation; sampled rows
    n, k = 131072, 4096
    t1, t2, a1, a2 = _planes(5, n, k, DEV)
    blocks = ops.pack_free(t1, t2, a1, a2, ws)
    del t1, t2
    x = inputs.hidden_states(6, 1, k)[0]
    q, da, bs = ops.quantize_act(x.to(DEV), ws)
    y = ops.gemv_free(blocks, n, k, q, da, bs, ws)
    B.tqfx4_check(ws)
    groups = np.unique(np.concatenate([np.arange(4), np.arange(n // 4 - 4, n // 4),
                                       np.random.default_rng(0).integers(0, n // 4, 100)]))
    rows = (groups[:, None] * 4 + np.arange(4)[None, :]).reshape(-1)
    # the oracle packs the sampled rows itself, from the same generated planes
    t1, t2, a1, a2 = _planes(5, n, k, DEV)
    ri = torch.from_numpy(rows).to(DEV)
    ref = oracle.pack_free(t1[ri].cpu().numpy(), t2[ri].cpu().numpy(), _np16(a1[ri]), _np16(a2[ri]))
    del t1, t2
    gb = B.tqfx4_free_bytes(4, k)
    sub = blocks.view(n // 4, gb)[torch.from_numpy(groups).to(DEV)].cpu().numpy().reshape(-1)
    assert np.array_equal(sub, ref)
    rq, rda, _ = oracle.quantize_act(x.numpy())
    assert np.array_equal(q.cpu().numpy(), rq)
    ry, _, _ = oracle.free_gemv(ref, 4 * len(groups), k, rq, rda)
    assert np.array_equal(y.cpu().numpy()[rows].view(np.uint32), ry.view(np.uint32))


def test_pack_reports_bad_trit_and_argument_errors(ws):
    n, k = 8, 512
    t1, t2, a1, a2 = _planes(7, n, k)
    t1[3, 300] = 2
    ops.pack_free(t1.to(DEV), t2.to(DEV), a1.to(DEV), a2.to(DEV), ws)
    with pytest.raises(B.TqfxError) as e:
        B.tqfx4_check(ws)
    assert e.value.status == 7
    y = torch.empty(n, device=DEV)
    blocks = torch.zeros(B.tqfx4_free_bytes(n, k) + 16, dtype=torch.uint8, device=DEV)
    q = torch.zeros(k, dtype=torch.int8, device=DEV)
    da = torch.ones(k // 256, device=DEV)
    bs = torch.zeros(k // 256, dtype=torch.int32, device=DEV)
    with pytest.raises(B.TqfxError) as e:  # n not a multiple of 4
        B.tqfx4_gemv_free(blocks, 6, k, q, da, bs, y, None, None, ws)
    assert e.value.status == 2
    with pytest.raises(B.TqfxError) as e:  # misaligned blocks
        B.tqfx4_gemv_free(blocks[1:], n, k, q, da, bs, y, None, None, ws)
    assert e.value.status == 3
    with pytest.raises(B.TqfxError) as e:  # S1 without S2
        B.tqfx4_gemv_free(blocks, n, k, q, da, bs, y, torch.empty(n * 2, dtype=torch.int32, device=DEV), None,
                          ws)
    assert e.value.status == 1
    B.tqfx4_gemv_free(blocks, 0, k, q, da, bs, y, None, None, ws)  # n = 0 is a no-op
    B.tqfx4_check(ws)
