"""ctypes/numpy wrapper around the plain-C tq2_0_fx4 oracle (tqfx4_oracle.c).

TEST INFRASTRUCTURE ONLY: the test suite, ``__graft_entry__.smoke()`` and the
CPU-baseline leg of ``bench.py`` are the only callers. The product path (the
CUDA library and its Python binding) never imports this package, and this
package never imports the product.

Each function restates the paper's arithmetic (Tied Trit-Planes, Sec. 2.1 and
2.2) through the C oracle; see the comments in tqfx4_oracle.c for the readings
taken where the paper is silent.
"""
import ctypes as C

import numpy as np

from .build_oracle import build as _build

QK = 256
ROWS = 4
BLOCK_BYTES = 520

_lib = None


def _p(a):
    return a.ctypes.data_as(C.c_void_p)


def lib():
    global _lib
    if _lib is None:
        path = _build()
        L = C.CDLL(path)
        i64, vp, i32 = C.c_int64, C.c_void_p, C.c_int
        sig = {
            "tqo_fold": (i32, [i32, i32]),
            "tqo_unfold": (i32, [i32, vp, vp]),
            "tqo_f32_to_f16": (C.c_uint16, [C.c_float]),
            "tqo_f16_to_f32": (C.c_float, [C.c_uint16]),
            "tqo_matrix_bytes": (i64, [i64, i64]),
            "tqo_pack_trits": (i32, [vp, vp, vp, i64, i64, vp]),
            "tqo_pack_rtn": (i32, [vp, i64, i64, vp]),
            "tqo_pack_tied": (i32, [vp, i64, i64, i32, vp, vp]),
            "tqo_mxfp4_bytes": (i64, [i64, i64]),
            "tqo_mxfp4_dequant": (i32, [vp, i64, i64, vp]),
            "tqo_mxfp4_gemv": (i32, [vp, i64, i64, vp, vp, vp, vp]),
            "tqo_free_bytes": (i64, [i64, i64]),
            "tqo_pack_free": (i32, [vp, vp, vp, vp, i64, i64, vp]),
            "tqo_free_dequant": (i32, [vp, i64, i64, vp]),
            "tqo_free_gemv": (i32, [vp, i64, i64, vp, vp, vp, vp, vp]),
            "tqo_expert_ffn_mxfp4": (i32, [vp, vp, vp, i64, i64, vp, vp, vp, vp, vp, vp, vp, vp]),
            "tqo_moe_tokens_fmt": (i32, [i32, vp, vp, vp, i64, i64, i64, vp, vp, i32, vp, i64, vp, vp, vp]),
            "tqo_unpack": (i32, [vp, i64, i64, vp, vp]),
            "tqo_dequant": (i32, [vp, i64, i64, vp]),
            "tqo_quantize_act": (i32, [vp, i64, i64, vp, vp, vp]),
            "tqo_block_sums": (i32, [vp, i64, i64, vp, vp]),
            "tqo_gemv": (i32, [vp, i64, i64, vp, vp, vp, vp]),
            "tqo_expf": (C.c_float, [C.c_float]),
            "tqo_swiglu": (None, [vp, vp, i64, vp]),
            "tqo_expert_ffn": (i32, [vp, vp, vp, i64, i64, vp, vp, vp, vp, vp, vp, vp, vp]),
            "tqo_router": (i32, [vp, vp, i64, i64, vp, i32, vp, vp, vp]),
            "tqo_moe_token": (i32, [vp, vp, vp, i64, i64, i64, vp, vp, i32, vp, vp, vp, vp]),
            "tqo_moe_tokens": (i32, [vp, vp, vp, i64, i64, i64, vp, vp, i32, vp, i64, vp, vp, vp]),
            "tqo_group_by_expert": (i32, [vp, i64, i32, i64, vp, vp, vp, vp]),
            "tqo_f32_to_f16_n": (None, [vp, i64, vp]),
            "tqo_f16_to_f32_n": (None, [vp, i64, vp]),
            "tqo_expf_n": (None, [vp, i64, vp]),
        }
        for name, (res, args) in sig.items():
            f = getattr(L, name)
            f.restype = res
            f.argtypes = args
        _lib = L
    return _lib


class OracleError(RuntimeError):
    pass


def _check(rc, what):
    if rc != 0:
        raise OracleError("%s failed with code %d" % (what, rc))


def _c(a, dt):
    return np.ascontiguousarray(a, dtype=dt)


# ---- Sec. 2.1: fold -------------------------------------------------------

def fold(t1: int, t2: int) -> int:
    return lib().tqo_fold(int(t1), int(t2))


def unfold(c: int):
    t1, t2 = C.c_int(), C.c_int()
    rc = lib().tqo_unfold(int(c), C.byref(t1), C.byref(t2))
    _check(rc, "unfold")
    return t1.value, t2.value


# ---- binary16 --------------------------------------------------------------

def f32_to_f16_bits(x) -> np.ndarray:
    x = _c(x, np.float32)
    out = np.empty(x.shape, np.uint16)
    lib().tqo_f32_to_f16_n(_p(x), x.size, _p(out))
    return out


def f16_bits_to_f32(h) -> np.ndarray:
    h = _c(h, np.uint16)
    out = np.empty(h.shape, np.float32)
    lib().tqo_f16_to_f32_n(_p(h), h.size, _p(out))
    return out


# ---- Sec. 2.2: format -------------------------------------------------------

def matrix_bytes(n: int, k: int) -> int:
    return int(lib().tqo_matrix_bytes(n, k))


def pack_rtn(w) -> np.ndarray:
    w = _c(w, np.float32)
    n, k = w.shape
    nbytes = matrix_bytes(n, k)
    if nbytes < 0:
        raise OracleError("bad shape %r" % (w.shape,))
    out = np.empty(nbytes, np.uint8)
    _check(lib().tqo_pack_rtn(_p(w), n, k, _p(out)), "pack_rtn")
    return out


def pack_tied(w, max_iter=64, with_iters=False):
    """The tied alternating solver (Sec. 2.1), see tqo_pack_tied: blocks, and
    with with_iters the scale updates per (row, block) (negated where
    max_iter stopped a block before its fixed point)."""
    w = _c(w, np.float32)
    n, k = w.shape
    nbytes = matrix_bytes(n, k)
    if nbytes < 0:
        raise OracleError("bad shape %r" % (w.shape,))
    out = np.empty(nbytes, np.uint8)
    iters = np.empty((n, k // 256), np.int32)
    _check(lib().tqo_pack_tied(_p(w), n, k, int(max_iter), _p(out), _p(iters)), "pack_tied")
    return (out, iters) if with_iters else out


def mxfp4_bytes(n: int, k: int) -> int:
    return int(lib().tqo_mxfp4_bytes(n, k))


def mxfp4_dequant(blocks, n: int, k: int) -> np.ndarray:
    """fp64 W [n][k] of MXFP4 blocks (17 bytes per 32 elements)."""
    blocks = _c(blocks, np.uint8)
    w = np.empty((n, k), np.float64)
    _check(lib().tqo_mxfp4_dequant(_p(blocks), n, k, _p(w)), "mxfp4_dequant")
    return w


def mxfp4_gemv(blocks, n: int, k: int, q, da):
    """(y fp32 [n], S int32 [n][k/32]) of the MXFP4 dot pass."""
    blocks = _c(blocks, np.uint8)
    q = _c(q, np.int8)
    da = _c(da, np.float32)
    y = np.empty(n, np.float32)
    S = np.empty((n, k // 32), np.int32)
    _check(lib().tqo_mxfp4_gemv(_p(blocks), n, k, _p(q), _p(da), _p(y), _p(S)), "mxfp4_gemv")
    return y, S


# ---- the free-scale two-plane format (Table 1, 4.125 bits/weight) ------------

def free_bytes(n: int, k: int) -> int:
    return int(lib().tqo_free_bytes(n, k))


def pack_free(t1, t2, a1_bits, a2_bits) -> np.ndarray:
    """Two trit planes int8 [n][k] and their f16 scale bits [n][k/256] ->
    528-byte blocks."""
    t1, t2 = _c(t1, np.int8), _c(t2, np.int8)
    a1_bits, a2_bits = _c(a1_bits, np.uint16), _c(a2_bits, np.uint16)
    n, k = t1.shape
    nbytes = free_bytes(n, k)
    if nbytes < 0:
        raise OracleError("bad shape %r" % (t1.shape,))
    out = np.empty(nbytes, np.uint8)
    _check(lib().tqo_pack_free(_p(t1), _p(t2), _p(a1_bits), _p(a2_bits), n, k, _p(out)), "pack_free")
    return out


def free_dequant(blocks, n: int, k: int) -> np.ndarray:
    blocks = _c(blocks, np.uint8)
    w = np.empty((n, k), np.float64)
    _check(lib().tqo_free_dequant(_p(blocks), n, k, _p(w)), "free_dequant")
    return w


def free_gemv(blocks, n: int, k: int, q, da):
    """(y fp32 [n], S1, S2 int32 [n][k/256]) of the two-plane dot pass."""
    blocks = _c(blocks, np.uint8)
    q, da = _c(q, np.int8), _c(da, np.float32)
    y = np.empty(n, np.float32)
    S1 = np.empty((n, k // QK), np.int32)
    S2 = np.empty((n, k // QK), np.int32)
    _check(lib().tqo_free_gemv(_p(blocks), n, k, _p(q), _p(da), _p(y), _p(S1), _p(S2)), "free_gemv")
    return y, S1, S2


def pack_trits(t1, t2, d_bits) -> np.ndarray:
    t1 = _c(t1, np.int8)
    t2 = _c(t2, np.int8)
    d_bits = _c(d_bits, np.uint16)
    n, k = t1.shape
    nbytes = matrix_bytes(n, k)
    if nbytes < 0:
        raise OracleError("bad shape %r" % (t1.shape,))
    out = np.empty(nbytes, np.uint8)
    _check(lib().tqo_pack_trits(_p(t1), _p(t2), _p(d_bits), n, k, _p(out)), "pack_trits")
    return out


def unpack(blocks, n: int, k: int):
    blocks = _c(blocks, np.uint8)
    c = np.empty((n, k), np.int8)
    d = np.empty((n, k // QK), np.uint16)
    _check(lib().tqo_unpack(_p(blocks), n, k, _p(c), _p(d)), "unpack")
    return c, d


def dequant(blocks, n: int, k: int) -> np.ndarray:
    blocks = _c(blocks, np.uint8)
    w = np.empty((n, k), np.float64)
    _check(lib().tqo_dequant(_p(blocks), n, k, _p(w)), "dequant")
    return w


# ---- Sec. 2.2: activations and the dot pass ------------------------------

def quantize_act(x):
    x = _c(x, np.float32)
    squeeze = x.ndim == 1
    if squeeze:
        x = x[None, :]
    m, k = x.shape
    q = np.empty((m, k), np.int8)
    da = np.empty((m, k // QK), np.float32)
    bs = np.empty((m, k // QK), np.int32)
    _check(lib().tqo_quantize_act(_p(x), m, k, _p(q), _p(da), _p(bs)), "quantize_act")
    if squeeze:
        return q[0], da[0], bs[0]
    return q, da, bs


def block_sums(blocks, n: int, k: int, q) -> np.ndarray:
    blocks = _c(blocks, np.uint8)
    q = _c(q, np.int8)
    S = np.empty((n, k // QK), np.int32)
    _check(lib().tqo_block_sums(_p(blocks), n, k, _p(q), _p(S)), "block_sums")
    return S


def gemv(blocks, n: int, k: int, q, da):
    blocks = _c(blocks, np.uint8)
    q = _c(q, np.int8)
    da = _c(da, np.float32)
    y = np.empty(n, np.float32)
    S = np.empty((n, k // QK), np.int32)
    _check(lib().tqo_gemv(_p(blocks), n, k, _p(q), _p(da), _p(y), _p(S)), "gemv")
    return y, S


def expf(z) -> np.ndarray:
    z = _c(z, np.float32)
    out = np.empty(z.shape, np.float32)
    lib().tqo_expf_n(_p(z), z.size, _p(out))
    return out


def swiglu(g, u) -> np.ndarray:
    g = _c(g, np.float32)
    u = _c(u, np.float32)
    h = np.empty(g.shape, np.float32)
    lib().tqo_swiglu(_p(g), _p(u), g.size, _p(h))
    return h


def expert_ffn(gate, up, down, hidden: int, inter: int, x, fmt: str = "fx4"):
    """One SwiGLU expert; returns (out, debug dict of g, u, h, qh, dh, bh).
    fmt: the weight format of gate, up and down ("fx4" or "mxfp4")."""
    gate, up, down = (_c(a, np.uint8) for a in (gate, up, down))
    x = _c(x, np.float32)
    out = np.empty(hidden, np.float32)
    g = np.empty(inter, np.float32)
    u = np.empty(inter, np.float32)
    h = np.empty(inter, np.float32)
    qh = np.empty(inter, np.int8)
    dh = np.empty(inter // QK, np.float32)
    bh = np.empty(inter // QK, np.int32)
    fn = {"fx4": lib().tqo_expert_ffn, "mxfp4": lib().tqo_expert_ffn_mxfp4}[fmt]
    _check(fn(_p(gate), _p(up), _p(down), hidden, inter, _p(x), _p(out),
              _p(g), _p(u), _p(h), _p(qh), _p(dh), _p(bh)), "expert_ffn")
    return out, dict(g=g, u=u, h=h, qh=qh, dh=dh, bh=bh)


# ---- router and MoE -----------------------------------------------------------

def router(Wr, bias, x, top_k: int):
    Wr = _c(Wr, np.float32)
    E, H = Wr.shape
    x = _c(x, np.float32)
    b = None if bias is None else _c(bias, np.float32)
    logits = np.empty(E, np.float64)
    idx = np.empty(top_k, np.int32)
    w = np.empty(top_k, np.float32)
    _check(lib().tqo_router(_p(Wr), None if b is None else _p(b), E, H, _p(x), top_k,
                            _p(logits), _p(idx), _p(w)), "router")
    return logits, idx, w


def _expert_ptrs(experts, E):
    """experts: dict e -> (gate_blocks, up_blocks, down_blocks) (numpy uint8)."""
    keep = []
    arrs = [(C.c_void_p * E)() for _ in range(3)]
    for e, trip in experts.items():
        for p, a in enumerate(trip):
            a = _c(a, np.uint8)
            keep.append(a)
            arrs[p][e] = a.ctypes.data
    return arrs, keep


def moe_tokens(experts, E: int, hidden: int, inter: int, Wr, bias, top_k: int, X, fmt: str = "fx4"):
    """Each token of X [T][hidden] through the MoE layer (per-token definition).

    experts: dict expert id -> (gate, up, down) block arrays in format fmt
    ("fx4" or "mxfp4"); experts a token does not select may be absent."""
    X = _c(X, np.float32)
    if X.ndim == 1:
        X = X[None, :]
    T = X.shape[0]
    Wr = _c(Wr, np.float32)
    b = None if bias is None else _c(bias, np.float32)
    (g, u, d), keep = _expert_ptrs(experts, E)
    OUT = np.empty((T, hidden), np.float32)
    idx = np.empty((T, top_k), np.int32)
    w = np.empty((T, top_k), np.float32)
    rc = lib().tqo_moe_tokens_fmt({"fx4": 0, "mxfp4": 1}[fmt], g, u, d, E, hidden, inter, _p(Wr),
                                  None if b is None else _p(b), top_k, _p(X), T, _p(OUT), _p(idx), _p(w))
    del keep
    _check(rc, "moe_tokens")
    return OUT, idx, w


def group_by_expert(idx, E: int):
    idx = _c(idx, np.int32)
    T, top_k = idx.shape
    counts = np.empty(E, np.int32)
    offsets = np.empty(E + 1, np.int32)
    pt = np.empty(T * top_k, np.int32)
    ps = np.empty(T * top_k, np.int32)
    _check(lib().tqo_group_by_expert(_p(idx), T, top_k, E, _p(counts), _p(offsets),
                                     _p(pt), _p(ps)), "group_by_expert")
    return counts, offsets, pt, ps
