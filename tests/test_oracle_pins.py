"""Pins of the CPU oracle against what the paper and the mathematics fix.

None of these tests re-types the oracle's formulas: each compares it with an
independent characterization (the paper's printed table and sizes, the
PTQTP two-plane form, brute-force argmin over the code alphabet, numpy's
binary16 and fp64 routines, library sorting), so that a dropped term, a
wrong sign or index, or a transposed operand in the oracle fails one of them.
"""
import os

import numpy as np
import pytest

import oracle

GOLD = os.path.join(os.path.dirname(__file__), "golden")


def _read_table(name):
    rows = []
    with open(os.path.join(GOLD, name)) as f:
        for line in f:
            line = line.split("#", 1)[0].strip()
            if line:
                rows.append(line.split())
    return rows


# ---------------------------------------------------------------- Sec. 2.1

def test_fold_table_matches_paper():
    rows = _read_table("fold_table.txt")
    assert len(rows) == 9
    codes = set()
    for t1, t2, c in rows:
        t1, t2, c = int(t1), int(t2), int(c)
        assert oracle.fold(t1, t2) == c
        assert oracle.unfold(c) == (t1, t2)
        codes.add(c)
    assert codes == set(range(-4, 5))  # a bijection onto the nine levels


def test_fold_rejects_non_trits():
    assert oracle.fold(2, 0) == -100
    assert oracle.fold(0, -2) == -100
    with pytest.raises(oracle.OracleError):
        oracle.unfold(5)


def test_ratio_three_is_the_only_uniform_nine_level_tie():
    # Sec. 2.1: ratios 1 and 2 give 5 and 7 uniformly spaced levels, ratio 3
    # gives nine uniformly spaced levels; other ratios give nine non-uniform.
    def levels(r):
        return sorted({r * a + b for a in (-1, 0, 1) for b in (-1, 0, 1)})

    def uniform(v):
        d = np.diff(v)
        return np.allclose(d, d[0])

    assert len(levels(1)) == 5 and uniform(levels(1))
    assert len(levels(2)) == 7 and uniform(levels(2))
    assert len(levels(3)) == 9 and uniform(levels(3))
    for r in (1.5, 2.5, 4, 5):
        lv = levels(r)
        assert len(lv) == 9 and not uniform(lv)


def test_fold_is_lossless_for_the_two_plane_form():
    # PTQTP writes W ~ a1 T1 + a2 T2 (Sec. 2.1); with a = (3s, s) the folded
    # block must dequantize to exactly that two-plane sum.
    rng = np.random.default_rng(1)
    n, k = 8, 512
    t1 = rng.integers(-1, 2, (n, k)).astype(np.int8)
    t2 = rng.integers(-1, 2, (n, k)).astype(np.int8)
    s = (np.abs(rng.standard_normal((n, k // 256))) * 0.01).astype(np.float16)
    blocks = oracle.pack_trits(t1, t2, s.view(np.uint16))
    w_hat = oracle.dequant(blocks, n, k)
    sf = np.repeat(s.astype(np.float64), 256, axis=1)
    two_plane = (3.0 * sf) * t1 + sf * t2
    assert np.array_equal(w_hat, two_plane)
    c, d = oracle.unpack(blocks, n, k)
    assert np.array_equal(d, s.view(np.uint16))
    # the dequantized values lie on the uniform grid s * {-4..4}
    ratio = np.divide(w_hat, sf, out=np.zeros_like(w_hat), where=sf != 0)
    assert np.array_equal(ratio, np.round(ratio)) and np.abs(ratio).max() <= 4


def test_pack_trits_rejects_bad_trit():
    t1 = np.zeros((4, 256), np.int8)
    t2 = np.zeros((4, 256), np.int8)
    t2[2, 17] = 2
    with pytest.raises(oracle.OracleError):
        oracle.pack_trits(t1, t2, np.zeros((4, 1), np.uint16))


# ---------------------------------------------------------------- Sec. 2.2

def test_sizes_printed_in_the_paper():
    g = {r[0]: float(r[1]) for r in _read_table("format_sizes.txt")}
    assert oracle.matrix_bytes(4, 256) == g["block_bytes"] == 520
    assert g["code_bytes"] + 2 * g["scale_count"] == g["block_bytes"]
    elems = g["columns_per_block"] * g["elements_per_column_block"]
    assert g["code_bytes"] * 2 == elems
    assert oracle.matrix_bytes(4, 256) * 8 / elems == g["bits_per_weight"]
    assert g["moe_layers"] * g["projections"] * g["experts_per_stack"] == g["expert_matrix_solves"]
    # 4096 x 2048 expert projections reproduce every size the paper prints:
    mats = g["expert_matrix_solves"]
    weights = mats * 4096 * 2048
    gib = 2.0 ** 30
    q4k = weights * g["q4k_bits_per_weight"] / 8 / gib
    assert round(q4k) == g["q4k_expert_payload_gib"]
    fx4_experts = mats * oracle.matrix_bytes(4096, 2048) / gib
    assert abs(fx4_experts - weights * g["bits_per_weight"] / 8 / gib) < 1e-9
    trunk = g["q4k_file_gib"] - q4k  # the non-expert part of the q4_k file
    assert abs((fx4_experts + trunk) - g["fx4_file_gib"]) < 0.06
    red = 100 * (1 - g["fx4_file_gib"] / g["q4k_file_gib"])
    assert abs(red - g["file_size_reduction_pct"]) < 0.05
    # gate/up (inter x hidden) and down (hidden x inter) have the same size
    assert oracle.matrix_bytes(2048, 4096) == oracle.matrix_bytes(4096, 2048) == 4259840


def test_matrix_bytes_rejects_bad_shapes():
    assert oracle.matrix_bytes(6, 256) == -1
    assert oracle.matrix_bytes(4, 100) == -1
    assert oracle.matrix_bytes(0, 0) == 0


def test_block_layout_hand_worked_example():
    rows = _read_table("block_example.txt")
    c = np.zeros((4, 256), np.int64)
    j = np.arange(256)
    c[0] = j % 9 - 4
    c[1] = 4
    c[2] = -4
    c[3, 0], c[3, 128], c[3, 255] = 1, -1, 3
    t1 = np.zeros_like(c)
    t2 = np.zeros_like(c)
    for r in range(4):
        for i in range(256):
            t1[r, i], t2[r, i] = oracle.unfold(int(c[r, i]))
    scales = np.array([[0x3C00], [0x4000], [0x3800], [0x0000]], np.uint16)
    blk = oracle.pack_trits(t1, t2, scales)
    assert blk.size == 520
    expected = {}
    for r in rows:
        if r[0] == "byte":
            expected[int(r[1])] = int(r[2], 16)
        elif r[0] == "fill":
            a, b = (int(x) for x in r[1].split(".."))
            for o in range(a, b + 1):
                expected[o] = int(r[2], 16)
    for o, v in expected.items():
        assert blk[o] == v, "byte %d: %#x != %#x" % (o, blk[o], v)
    cc, dd = oracle.unpack(blk, 4, 256)
    assert np.array_equal(cc, c) and np.array_equal(dd, scales)


def test_unpack_rejects_invalid_nibble():
    blk = oracle.pack_rtn(np.zeros((4, 256), np.float32))
    blk[8 + 5] = 0x49  # low nibble 9 is not a code
    with pytest.raises(oracle.OracleError):
        oracle.unpack(blk, 4, 256)


# --------------------------------------------------------------- binary16

def test_f16_to_f32_exhaustive_against_numpy():
    h = np.arange(1 << 16, dtype=np.uint32).astype(np.uint16)
    ours = oracle.f16_bits_to_f32(h)
    ref = h.view(np.float16).astype(np.float32)
    finite = np.isfinite(ref)
    assert np.array_equal(ours[finite].view(np.uint32), ref[finite].view(np.uint32))
    assert np.array_equal(np.isnan(ours), np.isnan(ref))
    assert np.array_equal(np.isinf(ours), np.isinf(ref))


def test_f32_to_f16_round_to_nearest_even_against_numpy():
    rng = np.random.default_rng(2)
    x = np.concatenate([
        (rng.standard_normal(400000) * 10.0 ** rng.integers(-9, 6, 400000)).astype(np.float32),
        # exact halfway points between adjacent f16 values (ties to even)
        (np.arange(-3000, 3000, dtype=np.float32) + 0.5) * np.float32(2.0 ** -10),
        (np.arange(0, 2048, dtype=np.float32) + 0.5) * np.float32(2.0 ** -24),  # subnormal ties
        np.array([65504, 65519.99, 65520, 1e6, -1e6, 2.0 ** -25, 2.0 ** -26, 0.0, -0.0,
                  5.96e-8, 3e-8], np.float32),
    ]).astype(np.float32)
    ours = oracle.f32_to_f16_bits(x)
    with np.errstate(over="ignore"):
        ref = x.astype(np.float16).view(np.uint16)
    assert np.array_equal(ours, ref)


# ------------------------------------------------------------ RTN codes

def _argmin_codes(w, dq):
    """Brute force over the nine-level alphabet: the code minimizing |w - dq c|
    (fp64), ties to the larger magnitude (half away from zero)."""
    cand = np.arange(-4, 5, dtype=np.float64)
    err = np.abs(w[..., None].astype(np.float64) - dq[..., None] * cand)
    best = err.min(axis=-1, keepdims=True)
    tie = np.isclose(err, best, rtol=0, atol=0)
    mag = np.where(tie, np.abs(cand), -1)
    # among exact ties prefer larger |c|; sign follows w
    pick = np.argmax(mag + (np.sign(cand) == np.sign(w[..., None])) * 0.5, axis=-1)
    return cand[pick]


def test_rtn_codes_are_the_nearest_level():
    rng = np.random.default_rng(3)
    n, k = 64, 1024
    w = (rng.standard_t(5, (n, k)) * 0.02).astype(np.float32)
    blocks = oracle.pack_rtn(w)
    c, d = oracle.unpack(blocks, n, k)
    wb = w.reshape(n, k // 256, 256)
    amax = np.abs(wb).max(axis=-1)
    d_ref = (amax / np.float32(4)).astype(np.float16)
    assert np.array_equal(d, d_ref.view(np.uint16))
    dq = np.repeat(d_ref.astype(np.float64), 256, axis=1)
    ref = _argmin_codes(w, dq)
    # x * (1/dq) in binary32 can only differ from the exact quotient at a
    # near-midpoint; everywhere else the code must be the brute-force one.
    ratio = w.astype(np.float64) / dq
    near = np.abs(np.abs(ratio - np.trunc(ratio)) - 0.5) < 1e-5
    assert np.array_equal(c[~near], ref[~near])
    assert np.abs(c.astype(np.int64) - ref).max() <= 1
    assert near.sum() < 20


def test_rtn_closed_cases():
    w = np.zeros((4, 512), np.float32)
    w[1, 7] = 0.3            # a single spike in block 0 of row 1
    w[2, 256:] = 0.25 * np.arange(-4, 4.5, 0.5, dtype=np.float32).repeat(16)[:256]
    w[3, :9] = np.array([-4, -3, -2, -1, 0, 1, 2, 3, 4], np.float32) * 0.5
    w[3, 9] = 1.25           # 2.5 * 0.5: a half tie goes away from zero -> 3
    w[3, 10] = -0.75         # -1.5 * 0.5 -> -2
    blocks = oracle.pack_rtn(w)
    c, d = oracle.unpack(blocks, 4, 512)
    assert d[0, 0] == 0 and not c[0].any()                       # zero block: d = 0, codes 0
    assert d[1, 0] == np.float16(0.3 / 4).view(np.uint16)
    assert c[1, 7] == 4 and np.count_nonzero(c[1]) == 1          # the spike is +4
    # block (2,1): amax = 1.0 -> d = 0.25; values k * 0.125 = half steps
    row = c[2, 256:].astype(np.int64)
    vals = w[2, 256:] / np.float32(0.25)
    assert np.array_equal(row, np.sign(vals) * np.floor(np.abs(vals) + 0.5))
    assert np.array_equal(c[3, :9], np.arange(-4, 5))            # exact multiples
    assert c[3, 9] == 3 and c[3, 10] == -2


def test_rtn_rejects_nonfinite():
    w = np.zeros((4, 256), np.float32)
    w[0, 0] = np.inf
    with pytest.raises(oracle.OracleError):
        oracle.pack_rtn(w)


# ------------------------------------------------- activation quantization

def test_quantize_act_nearest_level_and_sums():
    rng = np.random.default_rng(4)
    x = rng.standard_normal((5, 1024)).astype(np.float32) * np.float32(3.0)
    x[1, 256:512] = 0.0
    q, da, bs = oracle.quantize_act(x)
    xb = x.reshape(5, 4, 256)
    amax = np.abs(xb).max(axis=-1)
    assert np.array_equal(da, amax / np.float32(127))
    assert np.array_equal(bs, q.reshape(5, 4, 256).astype(np.int64).sum(-1))
    assert da[1, 1] == 0 and not q[1, 256:512].any()
    s = np.repeat(da.astype(np.float64), 256, axis=1)
    ratio = np.divide(x.astype(np.float64), s, out=np.zeros((5, 1024)), where=s != 0)
    exact = np.sign(ratio) * np.floor(np.abs(ratio) + 0.5)
    near = np.abs(np.abs(ratio - np.trunc(ratio)) - 0.5) < 1e-4
    assert np.array_equal(q[~near], np.clip(exact, -127, 127)[~near])
    # the absmax element of every nonzero block maps to +-127
    i = np.abs(xb).argmax(-1)
    qm = np.take_along_axis(q.reshape(5, 4, 256), i[..., None], -1)[..., 0]
    assert np.all((np.abs(qm) == 127) | (amax == 0))


# ----------------------------------------------------------- the dot pass

def test_block_sums_by_enumeration():
    rng = np.random.default_rng(5)
    n, k = 12, 768
    t1 = rng.integers(-1, 2, (n, k))
    t2 = rng.integers(-1, 2, (n, k))
    s = np.full((n, k // 256), 0x3C00, np.uint16)
    blocks = oracle.pack_trits(t1, t2, s)
    q = rng.integers(-127, 128, k).astype(np.int8)
    S = oracle.block_sums(blocks, n, k, q)
    c = 3 * t1 + t2  # the two-plane composite (Sec. 2.1) of the input planes
    ref = np.einsum("nbj,bj->nb", c.reshape(n, k // 256, 256), q.astype(np.int64).reshape(k // 256, 256))
    assert np.array_equal(S, ref)
    # extreme magnitudes stay exact: |S| <= 256 * 4 * 127
    blocks = oracle.pack_trits(np.ones((4, 256)), np.ones((4, 256)), np.full((4, 1), 0x3C00, np.uint16))
    S = oracle.block_sums(blocks, 4, 256, np.full(256, -127, np.int8))
    assert np.all(S == -130048)


def test_gemv_matches_fp64_brute_force():
    rng = np.random.default_rng(6)
    n, k = 64, 2048
    w = (rng.standard_normal((n, k)) * 0.02).astype(np.float32)
    x = rng.standard_normal(k).astype(np.float32)
    blocks = oracle.pack_rtn(w)
    q, da, bs = oracle.quantize_act(x)
    y, S = oracle.gemv(blocks, n, k, q, da)
    w_hat = oracle.dequant(blocks, n, k)
    x_hat = np.repeat(da.astype(np.float64), 256) * q
    ref = w_hat @ x_hat  # numpy fp64 matmul on dequantized operands
    terms = np.abs(w_hat) @ np.abs(x_hat)
    bound = (3 * (k // 256) + 2) * 2.0 ** -24 * terms
    assert np.all(np.abs(y - ref) <= bound)
    # and the quantized product tracks the fp32 product: nine levels per
    # absmax/4 step leave a normwise error near the paper's ~0.18 relative
    # reconstruction error (Sec. 2.1), far below a wrong sign or transpose
    yf = w.astype(np.float64) @ x.astype(np.float64)
    rel = np.linalg.norm(y - yf) / np.linalg.norm(yf)
    assert rel < 0.3


def test_gemv_closed_form_uniform_codes():
    n, k = 8, 1024
    one = np.ones((n, k))
    blocks = oracle.pack_trits(one, one, np.full((n, k // 256), 0x3800, np.uint16))  # c = 4, d = 0.5
    q = np.full(k, 3, np.int8)
    da = np.array([1.0, 2.0, 0.5, 0.25], np.float32)
    y, S = oracle.gemv(blocks, n, k, q, da)
    assert np.all(S == 4 * 3 * 256)
    assert np.all(y == np.float32(3072 * 0.5 * (1.0 + 2.0 + 0.5 + 0.25)))


def test_gemv_empty_k():
    y, S = oracle.gemv(np.zeros(0, np.uint8), 4, 0, np.zeros(0, np.int8), np.zeros(0, np.float32))
    assert np.all(y == 0)


# ------------------------------------------------------------ exp / SwiGLU

def test_expf_within_two_ulp_of_fp64():
    z = np.concatenate([np.linspace(-87, 88, 2_000_001, dtype=np.float32),
                        np.array([0.0, -0.0, 1e-8, -1e-8, 0.5, -0.5], np.float32)])
    ours = oracle.expf(z).astype(np.float64)
    ref = np.exp(z.astype(np.float64))
    ulp = np.spacing(ref.astype(np.float32)).astype(np.float64)
    assert np.max(np.abs(ours - ref) / ulp) <= 2.0
    assert oracle.expf(np.array([0.0], np.float32))[0] == 1.0


def test_expf_clamps_outside_the_normal_range():
    big = oracle.expf(np.array([200.0, -200.0, 88.0, -87.0], np.float32))
    assert big[0] == big[2] and big[1] == big[3] and np.isfinite(big).all()


def test_swiglu_against_fp64():
    rng = np.random.default_rng(7)
    g = (rng.standard_normal(100000) * 4).astype(np.float32)
    u = rng.standard_normal(100000).astype(np.float32)
    h = oracle.swiglu(g, u).astype(np.float64)
    gd = g.astype(np.float64)
    ref = gd / (1 + np.exp(-gd)) * u
    ulp = np.spacing(np.abs(ref).astype(np.float32)).astype(np.float64)
    assert np.max(np.abs(h - ref) / np.maximum(ulp, 1e-45)) <= 6
    # silu(0) = 0, silu large = identity, silu very negative -> 0
    h = oracle.swiglu(np.array([0.0, 100.0, -100.0], np.float32), np.ones(3, np.float32))
    assert h[0] == 0 and h[1] == 100.0 and abs(h[2]) < 1e-30


# ------------------------------------------------------------------ router

def test_router_against_numpy():
    rng = np.random.default_rng(8)
    E, H, k = 64, 512, 6
    Wr = (rng.standard_normal((E, H)) * 0.02).astype(np.float32)
    x = rng.standard_normal(H).astype(np.float32)
    bias = (-1.1 * np.log(np.arange(1, E + 1))).astype(np.float32)
    logits, idx, w = oracle.router(Wr, bias, x, k)
    ref = Wr.astype(np.float64) @ x.astype(np.float64) + bias
    assert np.allclose(logits, ref, rtol=1e-12, atol=1e-12)
    order = np.lexsort((np.arange(E), -ref))[:k]
    assert np.array_equal(idx, order)
    sel = ref[order]
    p = np.exp(sel - sel.max())
    assert np.allclose(w, p / p.sum(), rtol=1e-6)
    assert abs(w.astype(np.float64).sum() - 1) < 1e-6
    full = np.exp(ref - ref.max())
    full /= full.sum()
    assert np.allclose(w, full[order] / full[order].sum(), rtol=1e-6)


def test_router_ties_go_to_lower_index():
    E, H = 16, 256
    Wr = np.zeros((E, H), np.float32)
    bias = np.zeros(E, np.float32)
    bias[[3, 5, 9, 12]] = 1.0
    logits, idx, w = oracle.router(Wr, bias, np.ones(H, np.float32), 3)
    assert list(idx) == [3, 5, 9]
    assert np.allclose(w, 1 / 3)


# --------------------------------------------------------------------- MoE

def _experts(rng, E, hidden, inter):
    ex = {}
    for e in range(E):
        ex[e] = tuple(oracle.pack_rtn((rng.standard_t(5, shape) * 0.02).astype(np.float32))
                      for shape in ((inter, hidden), (inter, hidden), (hidden, inter)))
    return ex


def test_expert_ffn_tracks_fp64_reference():
    rng = np.random.default_rng(9)
    hidden, inter = 512, 768
    (g, u, d), = _experts(rng, 1, hidden, inter).values()
    x = rng.standard_normal(hidden).astype(np.float32)
    out, dbg = oracle.expert_ffn(g, u, d, hidden, inter, x)
    G, U, D = (oracle.dequant(b, *s) for b, s in ((g, (inter, hidden)), (u, (inter, hidden)),
                                                   (d, (hidden, inter))))
    xd = x.astype(np.float64)
    gg, uu = G @ xd, U @ xd
    ref = D @ (gg / (1 + np.exp(-gg)) * uu)
    assert np.abs(out - ref).max() < 0.03 * np.abs(ref).max()
    # swapping gate and up would not pass this
    bad = D @ (uu / (1 + np.exp(-uu)) * gg)
    assert np.abs(bad - ref).max() > 0.1 * np.abs(ref).max()
    assert np.array_equal(dbg["h"], oracle.swiglu(dbg["g"], dbg["u"]))


def test_moe_single_expert_reduces_to_the_ffn():
    rng = np.random.default_rng(10)
    hidden, inter = 256, 512
    ex = _experts(rng, 1, hidden, inter)
    Wr = (rng.standard_normal((1, hidden)) * 0.02).astype(np.float32)
    x = rng.standard_normal(hidden).astype(np.float32)
    out, idx, w = oracle.moe_tokens(ex, 1, hidden, inter, Wr, None, 1, x)
    ffn, _ = oracle.expert_ffn(*ex[0], hidden, inter, x)
    assert idx[0, 0] == 0 and w[0, 0] == 1.0
    assert np.array_equal(out[0], ffn)


def test_moe_identical_experts_are_routing_independent():
    rng = np.random.default_rng(11)
    hidden, inter, E = 256, 256, 8
    one = _experts(rng, 1, hidden, inter)[0]
    ex = {e: one for e in range(E)}
    Wr = (rng.standard_normal((E, hidden)) * 0.02).astype(np.float32)
    X = rng.standard_normal((3, hidden)).astype(np.float32)
    out, idx, w = oracle.moe_tokens(ex, E, hidden, inter, Wr, None, 4, X)
    for t in range(3):
        ffn, _ = oracle.expert_ffn(*one, hidden, inter, X[t])
        assert np.allclose(out[t], ffn, rtol=1e-5, atol=1e-6 * np.abs(ffn).max())


def test_moe_tracks_fp64_reference():
    rng = np.random.default_rng(12)
    hidden, inter, E, k = 256, 512, 16, 4
    ex = _experts(rng, E, hidden, inter)
    Wr = (rng.standard_normal((E, hidden)) * 0.02).astype(np.float32)
    X = rng.standard_normal((4, hidden)).astype(np.float32)
    out, idx, w = oracle.moe_tokens(ex, E, hidden, inter, Wr, None, k, X)
    for t in range(4):
        l = Wr.astype(np.float64) @ X[t].astype(np.float64)
        sel = np.lexsort((np.arange(E), -l))[:k]
        assert np.array_equal(idx[t], sel)
        p = np.exp(l[sel] - l[sel].max())
        p /= p.sum()
        ref = np.zeros(hidden)
        for j, e in enumerate(sel):
            G, U, D = (oracle.dequant(b, *s) for b, s in
                       ((ex[e][0], (inter, hidden)), (ex[e][1], (inter, hidden)), (ex[e][2], (hidden, inter))))
            gg, uu = G @ X[t], U @ X[t]
            ref += p[j] * (D @ (gg / (1 + np.exp(-gg)) * uu))
        assert np.abs(out[t] - ref).max() < 0.03 * np.abs(ref).max()


def test_moe_missing_selected_expert_is_an_error():
    rng = np.random.default_rng(13)
    ex = _experts(rng, 2, 256, 256)
    Wr = np.zeros((4, 256), np.float32)
    with pytest.raises(oracle.OracleError):
        oracle.moe_tokens(ex, 4, 256, 256, Wr, np.array([0, 0, 0, 1], np.float32), 1,
                          np.ones(256, np.float32))


def test_group_by_expert_is_a_stable_counting_sort():
    rng = np.random.default_rng(14)
    T, k, E = 37, 5, 11
    idx = np.stack([rng.permutation(E)[:k] for _ in range(T)]).astype(np.int32)
    counts, offsets, pt, ps = oracle.group_by_expert(idx, E)
    pairs = sorted(((int(idx[t, j]), t, j) for t in range(T) for j in range(k)))
    assert list(zip(pt, ps)) == [(t, j) for _, t, j in pairs]
    assert np.array_equal(counts, np.bincount(idx.ravel(), minlength=E))
    assert np.array_equal(offsets, np.concatenate([[0], np.cumsum(counts)]))
