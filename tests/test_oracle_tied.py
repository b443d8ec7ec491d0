"""Pins of the oracle's tied alternating solver (Sec. 2.1: the solver
alternates the trit planes against the single scale s of the tie (3s, s),
i.e. it fits W_hat = s * c with c in -4..4; scales serialize to f16).

Each test checks a property the mathematics fixes, computed independently of
the oracle's own arithmetic (numpy binary16 rounding, fp64 errors, brute force
over the code alphabet and over neighbouring f16 scales, a hand-solved case):
  * a hand-solved block (one outlier among ones) gives the least-squares
    scale rounded to f16 and the codes nearest to it;
  * every stored block is a fixed point: its codes are the nearest levels to
    its own f16 scale, and its scale is the best f16 value for its codes
    (no neighbouring f16 value gives a smaller squared error);
  * the squared error never exceeds the round-to-nearest fit's, and is
    smaller in total on heavy-tailed weights;
  * blocks the round-to-nearest fit already solves exactly are unchanged.
"""
import numpy as np
import pytest

import oracle
from paper_2608_08910_gb300 import inputs


def _decode(blocks, n, k):
    c, d = oracle.unpack(blocks, n, k)
    s = d.view(np.float16).astype(np.float64)  # [n][k/256] binary16 scales
    return c.astype(np.float64), s


def _block_err(w, c, s):
    n, k = w.shape
    r = (w.astype(np.float64) - c * np.repeat(s, 256, axis=1)).reshape(n, k // 256, 256)
    return (r * r).sum(axis=2)


def test_hand_solved_block():
    # w = (8, 1, ..., 1): round-to-nearest takes s = 8/4 = 2, codes (4, 1, ..., 1)
    # (1/2 rounds away from zero). For those codes the least-squares scale is
    # <w,c>/<c,c> = (32 + 255) / (16 + 255) = 287/271 = 1.0590..., whose
    # nearest binary16 value is 1 + 60/1024 = 1.05859375 (0x3C3C). Against it
    # 8 -> 7.56 -> 4 and 1 -> 0.945 -> 1: the same codes, so this is the fixed
    # point, reached after one scale update.
    w = np.ones((4, 256), np.float32)
    w[:, 0] = 8.0
    blocks, iters = oracle.pack_tied(w, with_iters=True)
    c, d = oracle.unpack(blocks, 4, 256)
    assert np.all(d == 0x3C3C)
    assert np.all(c[:, 0] == 4) and np.all(c[:, 1:] == 1)
    assert np.all(iters == 1)
    # and it beats round-to-nearest by more than an order of magnitude
    cr, sr = _decode(oracle.pack_rtn(w), 4, 256)
    ct, st = _decode(blocks, 4, 256)
    assert _block_err(w, ct, st)[0, 0] < _block_err(w, cr, sr)[0, 0] / 10


@pytest.fixture(scope="module")
def heavy():
    # Student-t(5) * 0.02, the weights the benchmark layers use
    w = inputs.student_t((64, 2048), 5, 0.02, seed=11).numpy()
    blocks, iters = oracle.pack_tied(w, with_iters=True)
    return w, blocks, iters


def test_every_block_is_a_fixed_point(heavy):
    w, blocks, iters = heavy
    n, k = w.shape
    assert np.all(iters >= 0)  # no block stopped by the iteration cap
    c, s = _decode(blocks, n, k)
    # codes: the nearest level to w / s (brute force over -4..4; a tie at
    # exactly half a step is broken away from zero, as round-to-nearest does)
    sf = np.repeat(s, 256, axis=1)
    levels = np.arange(-4, 5, dtype=np.float64)
    dist = np.abs(w.astype(np.float64)[..., None] - sf[..., None] * levels)
    best = dist.min(axis=-1)
    mine = np.abs(w.astype(np.float64) - sf * c)
    assert np.all(mine <= best * (1 + 1e-6) + 1e-30)
    # scale: no neighbouring binary16 value fits these codes better
    err = _block_err(w, c, s)
    bits = s.astype(np.float16).view(np.uint16)
    for step in (-1, 1):
        nb16 = (bits.astype(np.int32) + step).clip(0, 0x7BFF).astype(np.uint16).view(np.float16).astype(np.float64)
        other = _block_err(w, c, nb16)
        assert np.all(err <= other * (1 + 1e-9))


def test_error_never_above_round_to_nearest(heavy):
    w, blocks, _ = heavy
    n, k = w.shape
    ct, st = _decode(blocks, n, k)
    cr, sr = _decode(oracle.pack_rtn(w), n, k)
    et, er = _block_err(w, ct, st), _block_err(w, cr, sr)
    assert np.all(et <= er * (1 + 1e-9))
    assert et.sum() < 0.9 * er.sum()  # heavy tails: the outlier-set scale is far from optimal


def test_exact_grid_blocks_are_unchanged():
    # blocks that are exactly s * c with an f16 scale s and a code of +-4 in
    # every block: round-to-nearest reproduces them exactly, so does the solver
    rng = np.random.default_rng(3)
    s = np.float16(0.01171875).astype(np.float32)  # a binary16 value
    c = rng.integers(-4, 5, size=(8, 512)).astype(np.float32)
    c[:, 0] = 4
    c[:, 256] = -4
    w = (s * c).astype(np.float32)
    bt, it = oracle.pack_tied(w, with_iters=True)
    assert np.array_equal(bt, oracle.pack_rtn(w))
    assert np.all(it == 0)


def test_zero_block_and_errors():
    w = np.zeros((4, 256), np.float32)
    bt, it = oracle.pack_tied(w, with_iters=True)
    assert np.array_equal(bt, oracle.pack_rtn(w)) and np.all(it == 0)
    w[1, 5] = np.inf
    with pytest.raises(oracle.OracleError):
        oracle.pack_tied(w)
    with pytest.raises(oracle.OracleError):
        oracle.pack_tied(np.zeros((3, 256), np.float32))


def test_deterministic_and_capped(heavy):
    w, blocks, iters = heavy
    assert np.array_equal(oracle.pack_tied(w), blocks)
    # with no update allowed the solver is round-to-nearest
    assert np.array_equal(oracle.pack_tied(w, max_iter=0), oracle.pack_rtn(w))
    assert iters.max() >= 2  # some blocks need several updates
