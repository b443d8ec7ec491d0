"""Pins of the oracle's free-scale two-plane format (Table 1's free-scale
K=2 row: two trit planes with two independent f16 scales per row and 256
columns, stored apart at 4.125 bits/weight because the pair does not fold).

Independent characterizations: the size printed in Table 1; a hand-built
block for the byte order; W = a1 t1 + a2 t2 built with numpy's float16;
exact plane sums by numpy; the dot pass against fp64 within the binary32
rounding of its schedule; and the tied special case a = (3s, s), where the
two planes must give the folded tq2_0_fx4 code's block sums exactly
(3 S1 + S2 = S) and the same output within rounding.
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2608_08910_gb300 import inputs


def _planes(seed, n, k):
    t1, t2, s = inputs.trit_planes(seed, n, k)
    s2 = inputs.trit_planes(seed + 1, n, k)[2]
    return t1.numpy(), t2.numpy(), s.view(torch.int16).numpy().view(np.uint16), \
        s2.view(torch.int16).numpy().view(np.uint16)


def test_size_is_4_125_bits_per_weight():
    assert oracle.free_bytes(1024, 1024) * 8 / (1024 * 1024) == 4.125
    assert oracle.free_bytes(6, 256) < 0 and oracle.free_bytes(4, 100) < 0


def test_hand_built_block():
    n, k = 4, 256
    t1 = np.zeros((n, k), np.int8)
    t2 = np.zeros((n, k), np.int8)
    t1[2, 5] = 1
    t2[1, 255] = -1
    a1 = np.zeros((n, 1), np.uint16)
    a2 = np.zeros((n, 1), np.uint16)
    a1[3, 0] = 0x3C00  # 1.0
    a2[0, 0] = 0xC000  # -2.0
    blk = oracle.pack_free(t1, t2, a1, a2)
    assert blk.size == 528
    assert blk[6] == 0x00 and blk[7] == 0x3C and blk[8] == 0x00 and blk[9] == 0xC0
    # every trit 0 is u = 1: 0b01 in each 2-bit field
    assert blk[16 + 128 * 2 + 1] == 0x59       # row 2, t1 element 5: u = 2 in bits 2..3
    assert blk[16 + 128 * 1 + 64 + 63] == 0x15  # row 1, t2 element 255: u = 0 in bits 6..7
    planes = np.delete(blk[16:], [128 * 2 + 1, 128 + 64 + 63])
    assert np.all(planes == 0x55)


def test_dequant_is_the_two_plane_sum():
    n, k = 8, 512
    t1, t2, a1, a2 = _planes(3, n, k)
    w = oracle.free_dequant(oracle.pack_free(t1, t2, a1, a2), n, k)
    s1 = np.repeat(a1.view(np.float16).astype(np.float64), 256, axis=1)
    s2 = np.repeat(a2.view(np.float16).astype(np.float64), 256, axis=1)
    assert np.array_equal(w, s1 * t1 + s2 * t2)


def test_invalid_trits_are_rejected():
    t1 = np.zeros((4, 256), np.int8)
    t1[0, 0] = 2
    with pytest.raises(oracle.OracleError):
        oracle.pack_free(t1, t1 * 0, np.zeros((4, 1), np.uint16), np.zeros((4, 1), np.uint16))
    blk = oracle.pack_free(t1 * 0, t1 * 0, np.zeros((4, 1), np.uint16), np.zeros((4, 1), np.uint16))
    blk[16] |= 3  # u = 3 in row 0, element 0
    with pytest.raises(oracle.OracleError):
        oracle.free_dequant(blk, 4, 256)
    with pytest.raises(oracle.OracleError):
        oracle.free_gemv(blk, 4, 256, np.zeros(256, np.int8), np.ones(1, np.float32))


@pytest.mark.parametrize("n,k", [(4, 256), (12, 1024), (40, 256 * 7)])
def test_gemv_sums_exact_and_output_within_rounding(n, k):
    t1, t2, a1, a2 = _planes(n + k, n, k)
    blocks = oracle.pack_free(t1, t2, a1, a2)
    x = inputs.hidden_states(k, 1, k)[0].numpy()
    q, da, _ = oracle.quantize_act(x)
    y, S1, S2 = oracle.free_gemv(blocks, n, k, q, da)
    qq = q.astype(np.int64)
    assert np.array_equal(S1, (t1.astype(np.int64) * qq).reshape(n, k // 256, 256).sum(axis=2))
    assert np.array_equal(S2, (t2.astype(np.int64) * qq).reshape(n, k // 256, 256).sum(axis=2))
    W = oracle.free_dequant(blocks, n, k)
    xa = qq * np.repeat(da.astype(np.float64), 256)
    terms = W * xa[None, :]
    exact = terms.sum(axis=1)
    # per block: two products, their sum, the running sum (plus the scale products)
    bound = 6 * (k // 256 + 1) * 2.0 ** -24 * np.abs(terms).sum(axis=1)
    assert np.all(np.abs(y.astype(np.float64) - exact) <= bound)


def test_tied_scales_reduce_to_the_folded_code():
    # a = (3s, s) with s of few mantissa bits, so that 3s is exact in f16
    n, k = 8, 1024
    t1, t2, _, _ = _planes(9, n, k)
    rng = np.random.default_rng(9)
    s = (rng.integers(1, 64, (n, k // 256)) * 2.0 ** -12).astype(np.float16)
    a1 = (3 * s.astype(np.float32)).astype(np.float16)
    assert np.array_equal(a1.astype(np.float64), 3 * s.astype(np.float64))
    free = oracle.pack_free(t1, t2, a1.view(np.uint16), s.view(np.uint16))
    fx4 = oracle.pack_trits(t1, t2, s.view(np.uint16))
    x = inputs.hidden_states(10, 1, k)[0].numpy()
    q, da, _ = oracle.quantize_act(x)
    y, S1, S2 = oracle.free_gemv(free, n, k, q, da)
    yf, S = oracle.gemv(fx4, n, k, q, da)
    assert np.array_equal(3 * S1 + S2, S)
    assert np.array_equal(oracle.free_dequant(free, n, k), oracle.dequant(fx4, n, k))
    assert np.allclose(y, yf, rtol=1e-5, atol=1e-5 * np.abs(yf).max())
