"""Pins of the oracle's MXFP4 arm (the released expert bytes of Sec. 2.3, Table 1's
4.25-bit format, served directly by an integer dot pass).

Independent characterizations: the OCP microscaling definition of e2m1 from
its bit fields (sign, 2-bit exponent with bias 1, 1-bit mantissa, a
subnormal at exponent 0) and of e8m0 (2^(E-127)), instead of the oracle's
doubled-code table; exact block sums by numpy enumeration; the dot pass
against an fp64 brute-force sum within the binary32 rounding of its
schedule; the byte order on a hand-built block.
"""
import numpy as np
import pytest

import oracle
from paper_2608_08910_gb300 import inputs


def _e2m1(nib):
    """OCP e2m1 value of a 4-bit code, from its bit fields."""
    nib = np.asarray(nib, dtype=np.int64)
    s = np.where(nib & 8, -1.0, 1.0)
    e = (nib >> 1) & 3
    m = nib & 1
    mag = np.where(e == 0, 0.5 * m, np.ldexp(1.0 + 0.5 * m, e - 1))
    return s * mag


def _ref_decode(blocks, n, k):
    """W [n][k] from the OCP definitions and the stated byte order."""
    b = np.asarray(blocks, np.uint8).reshape(n, k // 32, 17).astype(np.int64)
    scale = np.ldexp(1.0, b[..., 0] - 127)  # e8m0
    lo, hi = b[..., 1:] & 15, b[..., 1:] >> 4
    nib = np.concatenate([lo, hi], axis=-1)  # elements 0..15, then 16..31
    return (_e2m1(nib) * scale[..., None]).reshape(n, k), nib.reshape(n, k)


def test_size_is_4_25_bits_per_weight():
    # Table 1 lists the released MXFP4 bytes at 4.25 bits/weight
    assert oracle.mxfp4_bytes(1024, 1024) * 8 / (1024 * 1024) == 4.25
    assert oracle.mxfp4_bytes(4, 100) < 0


def test_e2m1_alphabet():
    # the eight magnitudes of e2m1 are those the doubled codes halve
    assert list(_e2m1(np.arange(8))) == [0.0, 0.5, 1.0, 1.5, 2.0, 3.0, 4.0, 6.0]


def test_hand_built_block():
    blk = np.zeros(17, np.uint8)
    blk[0] = 127          # scale 2^0
    blk[1] = 0x5A         # element 0: code 0xA (-1.0); element 16: code 0x5 (3.0)
    blk[16] = 0x7F        # element 15: code 0xF (-6.0); element 31: code 0x7 (6.0)
    w = oracle.mxfp4_dequant(blk, 1, 32)[0]
    assert w[0] == -1.0 and w[16] == 3.0 and w[15] == -6.0 and w[31] == 6.0
    assert np.count_nonzero(w) == 4
    blk[0] = 255          # NaN scale
    with pytest.raises(oracle.OracleError):
        oracle.mxfp4_dequant(blk, 1, 32)


@pytest.mark.parametrize("n,k", [(4, 256), (16, 1024), (12, 512 * 3)])
def test_dequant_matches_the_ocp_definition(n, k):
    blocks = inputs.mxfp4_matrix(n + k, n, k).numpy()
    ref, _ = _ref_decode(blocks, n, k)
    assert np.array_equal(oracle.mxfp4_dequant(blocks, n, k), ref)


@pytest.mark.parametrize("n,k", [(8, 256), (32, 2048)])
def test_gemv_against_brute_force(n, k):
    blocks = inputs.mxfp4_matrix(3 * n + k, n, k).numpy()
    x = inputs.hidden_states(n * 5 + k, 1, k)[0].numpy()
    q, da, _ = oracle.quantize_act(x)
    y, S = oracle.mxfp4_gemv(blocks, n, k, q, da)
    W, nib = _ref_decode(blocks, n, k)
    # exact block sums: S = sum over the block of (2 * e2m1) * q
    c = (2.0 * _e2m1(nib)).astype(np.int64)
    S_ref = (c * q.astype(np.int64)[None, :]).reshape(n, k // 32, 32).sum(axis=2)
    assert np.array_equal(S, S_ref)
    # the dot pass equals the fp64 dot product of the dequantized operands,
    # within the schedule's binary32 roundings (one per block product and sum)
    xa = q.astype(np.float64) * np.repeat(da.astype(np.float64), 256)
    terms = W * xa[None, :]
    exact = terms.sum(axis=1)
    bound = 2 * (k // 32 + 1) * 2.0 ** -24 * np.abs(terms).sum(axis=1)
    assert np.all(np.abs(y.astype(np.float64) - exact) <= bound)


def _mx_expert(seed, hidden, inter):
    return tuple(inputs.mxfp4_matrix(seed * 3 + p, *shape).numpy()
                 for p, shape in enumerate(((inter, hidden), (inter, hidden), (hidden, inter))))


def test_mxfp4_expert_ffn_tracks_fp64_reference():
    # the SwiGLU expert over MXFP4 projections, against fp64 on the OCP-decoded weights
    hidden, inter = 512, 768
    g, u, d = _mx_expert(3, hidden, inter)
    x = inputs.hidden_states(4, 1, hidden)[0].numpy()
    out, dbg = oracle.expert_ffn(g, u, d, hidden, inter, x, fmt="mxfp4")
    G, _ = _ref_decode(g, inter, hidden)
    U, _ = _ref_decode(u, inter, hidden)
    D, _ = _ref_decode(d, hidden, inter)
    xd = x.astype(np.float64)
    gg, uu = G @ xd, U @ xd
    ref = D @ (gg / (1 + np.exp(-gg)) * uu)
    assert np.abs(out - ref).max() < 0.03 * np.abs(ref).max()
    bad = D @ (uu / (1 + np.exp(-uu)) * gg)  # gate and up swapped
    assert np.abs(bad - ref).max() > 0.1 * np.abs(ref).max()
    # the projections are the MXFP4 dot pass
    q, da, _ = oracle.quantize_act(x)
    assert np.array_equal(dbg["g"], oracle.mxfp4_gemv(g, inter, hidden, q, da)[0])


def test_mxfp4_moe_tracks_fp64_reference():
    hidden, inter, E, k = 512, 512, 8, 3
    ex = {e: _mx_expert(10 + e, hidden, inter) for e in range(E)}
    Wr = inputs.router_weight(5, E, hidden).numpy()
    X = inputs.hidden_states(6, 3, hidden).numpy()
    out, idx, w = oracle.moe_tokens(ex, E, hidden, inter, Wr, None, k, X, fmt="mxfp4")
    for t in range(3):
        l = Wr.astype(np.float64) @ X[t].astype(np.float64)
        sel = np.lexsort((np.arange(E), -l))[:k]
        assert np.array_equal(idx[t], sel)
        p = np.exp(l[sel] - l[sel].max())
        p /= p.sum()
        ref = np.zeros(hidden)
        for j, e in enumerate(sel):
            G, _ = _ref_decode(ex[e][0], inter, hidden)
            U, _ = _ref_decode(ex[e][1], inter, hidden)
            D, _ = _ref_decode(ex[e][2], hidden, inter)
            gg, uu = G @ X[t], U @ X[t]
            ref += p[j] * (D @ (gg / (1 + np.exp(-gg)) * uu))
        assert np.abs(out[t] - ref).max() < 0.03 * np.abs(ref).max()


def test_mxfp4_moe_single_expert_reduces_to_the_ffn():
    hidden, inter = 512, 512
    ex = {0: _mx_expert(30, hidden, inter)}
    Wr = np.zeros((1, hidden), np.float32)
    x = inputs.hidden_states(31, 1, hidden)[0].numpy()
    out, idx, w = oracle.moe_tokens(ex, 1, hidden, inter, Wr, None, 1, x, fmt="mxfp4")
    ffn, _ = oracle.expert_ffn(*ex[0], hidden, inter, x, fmt="mxfp4")
    assert idx[0, 0] == 0 and w[0, 0] == 1.0
    assert np.array_equal(out[0], ffn)
