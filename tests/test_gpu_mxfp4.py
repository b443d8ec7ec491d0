"""GPU parity of tqfx4_gemv_mxfp4 (the MXFP4 arm: released expert bytes,
17 bytes per 32 elements, served by the integer dot pass) against the CPU
oracle, through the C ABI: int32 block sums bit-exact, fp32 outputs bit-exact
(both sides run the same binary32 schedule: the exact block values of a
256-element activation group added in block order, each group sum times its
activation scale added in group order)."""
import numpy as np
import pytest
import torch

import oracle
from paper_2608_08910_gb300 import binding as B
from paper_2608_08910_gb300 import inputs, ops
from tests.parity import FP32_TOL, rel_err

pytestmark = pytest.mark.gpu
DEV = "cuda"

# expert gate/up (2048 x 4096) and down (4096 x 2048) shapes, a single row,
# rows not a multiple of the 16 rows a CTA starts with, odd block counts per
# lane (k/32 not a multiple of 32), the largest k
SHAPES = [(1, 512), (2048, 4096), (4096, 2048), (13, 1536), (300, 2560), (37, 7168), (1000, 512),
          (5, B.TQFX4_MAX_K)]


@pytest.fixture(scope="module")
def ws():
    return ops.workspace(B.TQFX4_STATUS_BYTES)


def _case(n, k, seed):
    blocks = inputs.mxfp4_matrix(seed, n, k)
    x = inputs.hidden_states(seed + 1, 1, k)[0]
    q, da, _ = oracle.quantize_act(x.numpy())
    return blocks, q, da


@pytest.mark.parametrize("n,k", SHAPES)
def test_gemv_mxfp4_bit_exact(n, k, ws):
    blocks, q, da = _case(n, k, 3 * n + k)
    ry, rS = oracle.mxfp4_gemv(blocks.numpy(), n, k, q, da)
    y, S = ops.gemv_mxfp4(blocks.to(DEV), n, k, torch.from_numpy(q).to(DEV), torch.from_numpy(da).to(DEV), ws,
                          block_sums=True)
    B.tqfx4_check(ws)
    assert np.array_equal(S.cpu().numpy(), rS)
    got = y.cpu().numpy()
    assert np.array_equal(got.view(np.uint32), ry.view(np.uint32))
    assert rel_err(got, ry) <= FP32_TOL


# without block sums (the kernel variant that skips them): rows not a
# multiple of the 16 rows a CTA starts with, k from one to 32 units of 512,
# and the largest k
TC_SHAPES = [(1, 512), (128, 512), (300, 1536), (2048, 4096), (4096, 2048), (1000, 8192), (5, 16384)]


@pytest.mark.parametrize("n,k", TC_SHAPES)
def test_gemv_mxfp4_without_sums_bit_exact(n, k, ws):
    blocks, q, da = _case(n, k, 7 * n + k)
    ry, _ = oracle.mxfp4_gemv(blocks.numpy(), n, k, q, da)
    y = ops.gemv_mxfp4(blocks.to(DEV), n, k, torch.from_numpy(q).to(DEV), torch.from_numpy(da).to(DEV), ws)
    B.tqfx4_check(ws)
    assert np.array_equal(y.cpu().numpy().view(np.uint32), ry.view(np.uint32))


def test_gemv_mxfp4_uses_device_quantized_activation(ws):
    # the activation from the library's own quantizer, as the decode path feeds it
    n, k = 512, 4096
    blocks = inputs.mxfp4_matrix(11, n, k)
    x = inputs.hidden_states(12, 1, k)[0]
    q, da, _ = ops.quantize_act(x.to(DEV), ws)
    y = ops.gemv_mxfp4(blocks.to(DEV), n, k, q, da, ws)
    B.tqfx4_check(ws)
    rq, rda, _ = oracle.quantize_act(x.numpy())  # the oracle quantizes its own copy
    assert np.array_equal(q.cpu().numpy(), rq) and np.array_equal(da.cpu().numpy().view(np.uint32),
                                                                  rda.view(np.uint32))
    ry, _ = oracle.mxfp4_gemv(blocks.numpy(), n, k, rq, rda)
    assert np.array_equal(y.cpu().numpy().view(np.uint32), ry.view(np.uint32))


def test_gemv_mxfp4_large_sampled(ws):
    # 131072 x 4096 (285 MB of blocks, larger than L2): sampled rows against the oracle
    n, k = 131072, 4096
    blocks = inputs.mxfp4_matrix(5, n, k, DEV)
    x = inputs.hidden_states(6, 1, k)[0]
    q, da, _ = oracle.quantize_act(x.numpy())
    y = ops.gemv_mxfp4(blocks, n, k, torch.from_numpy(q).to(DEV), torch.from_numpy(da).to(DEV), ws)
    B.tqfx4_check(ws)
    rows = np.unique(np.concatenate([np.arange(16), np.arange(n - 16, n),
                                     np.random.default_rng(0).integers(0, n, 200)]))
    rb = B.tqfx4_mxfp4_bytes(1, k)
    sub = blocks.view(n, rb)[torch.from_numpy(rows).to(DEV)].cpu().numpy()
    ry, _ = oracle.mxfp4_gemv(sub, len(rows), k, q, da)
    assert np.array_equal(y.cpu().numpy()[rows].view(np.uint32), ry.view(np.uint32))


def test_gemv_mxfp4_extreme_scales(ws):
    # E = 0 (2^-127, subnormal products) and E = 254 (2^127) next to ordinary blocks
    n, k = 64, 1024
    blocks = inputs.mxfp4_matrix(21, n, k).numpy().reshape(n, k // 32, 17).copy()
    blocks[::3, ::5, 0] = 0
    blocks[1::7, 2::9, 0] = 150
    blocks = blocks.reshape(-1)
    _, q, da = _case(n, k, 22)
    ry, rS = oracle.mxfp4_gemv(blocks, n, k, q, da)
    y, S = ops.gemv_mxfp4(torch.from_numpy(blocks).to(DEV), n, k, torch.from_numpy(q).to(DEV),
                          torch.from_numpy(da).to(DEV), ws, block_sums=True)
    B.tqfx4_check(ws)
    assert np.array_equal(S.cpu().numpy(), rS)
    assert np.array_equal(y.cpu().numpy().view(np.uint32), ry.view(np.uint32))


def test_gemv_mxfp4_nan_scale_and_argument_errors(ws):
    n, k = 8, 512
    blocks, q, da = _case(n, k, 31)
    bad = blocks.clone()
    bad[17 * 20] = 255  # block 4 of row 1: a NaN scale
    qd, dd = torch.from_numpy(q).to(DEV), torch.from_numpy(da).to(DEV)
    ops.gemv_mxfp4(bad.to(DEV), n, k, qd, dd, ws)
    with pytest.raises(B.TqfxError) as e:
        B.tqfx4_check(ws)
    assert e.value.status == 7
    y = torch.empty(n, device=DEV)
    with pytest.raises(B.TqfxError) as e:  # k not a multiple of 512
        B.tqfx4_gemv_mxfp4(blocks.to(DEV), n, 256, qd, dd, y, None, ws)
    assert e.value.status == 2
    with pytest.raises(B.TqfxError) as e:  # misaligned blocks
        B.tqfx4_gemv_mxfp4(torch.zeros(17 * 16 * n + 16, dtype=torch.uint8, device=DEV)[1:], n, k, qd, dd, y,
                           None, ws)
    assert e.value.status == 3
    with pytest.raises(B.TqfxError) as e:
        B.tqfx4_gemv_mxfp4(None, n, k, qd, dd, y, None, ws)
    assert e.value.status == 1
    # n = 0 is a no-op
    B.tqfx4_gemv_mxfp4(blocks.to(DEV), 0, k, qd, dd, y, None, ws)
    B.tqfx4_check(ws)
