"""ctypes binding of libtqfx4 (include/tqfx4.h), with the same names.

Argument marshalling only: torch tensors are passed as raw device pointers
with the caller's current CUDA stream; every step of the computation runs in
the library's CUDA kernels. There is no CPU fallback: if libtqfx4.so is
missing or a call fails, an exception is raised.
"""
import ctypes as C
import os

import torch

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "libtqfx4.so")
DEBUG_LIB_PATH = os.path.join(_HERE, "libtqfx4_debug.so")  # the TQFX4_DEBUG build (build.build(debug=True))

TQFX4_QK = 256
TQFX4_ROWS = 4
TQFX4_BLOCK_BYTES = 520
TQFX4_STATUS_BYTES = 256
TQFX4_MAX_K = 16384
TQFX4_NOALLOC_SCRATCH_BYTES = 1 << 20
TQFX4_SRC_TRITS = 0
TQFX4_SRC_F32_RTN = 1
TQFX4_SRC_F32_TIED = 2
TQFX4_TIED_MAX_ITER = 64
TQFX4_PATH_AUTO = 0
TQFX4_PATH_DECODE = 1
TQFX4_PATH_PREFILL = 2

STATUS_NAMES = {0: "TQFX4_OK", 1: "TQFX4_EINVAL", 2: "TQFX4_ESHAPE", 3: "TQFX4_EALIGN",
                4: "TQFX4_EWORKSPACE", 5: "TQFX4_ECUDA", 6: "TQFX4_ETIMEOUT", 7: "TQFX4_EDATA"}

_i64, _vp, _int, _sz = C.c_int64, C.c_void_p, C.c_int, C.c_size_t


class TqfxError(RuntimeError):
    def __init__(self, status, fn, msg):
        super().__init__("%s -> %s: %s" % (fn, STATUS_NAMES.get(status, status), msg))
        self.status = status


class CExperts(C.Structure):
    _fields_ = [("gate", _vp), ("up", _vp), ("down", _vp),
                ("n_experts", _i64), ("hidden", _i64), ("inter", _i64)]


class CRouter(C.Structure):
    _fields_ = [("weight", _vp), ("bias", _vp), ("top_k", C.c_int32)]


class CMoeViews(C.Structure):
    _fields_ = [(n, _sz) for n in ("logits", "logits_lo", "qx", "dx", "bx", "g", "u", "h", "qh", "dh", "bh", "o",
                                   "counts", "offsets", "pair_token", "pair_slot", "pair_of")]


_SIGS = {
    "tqfx4_matrix_bytes": (_i64, [_i64, _i64]),
    "tqfx4_basic_workspace_bytes": (_sz, []),
    "tqfx4_pack": (_int, [_int, _vp, _vp, _vp, _i64, _i64, _vp, _vp, _sz, _vp]),
    "tqfx4_quantize_act": (_int, [_vp, _i64, _i64, _vp, _vp, _vp, _vp, _sz, _vp]),
    "tqfx4_gemv": (_int, [_vp, _i64, _i64, _vp, _vp, _vp, _vp, _vp, _vp, _sz, _vp]),
    "tqfx4_gemv_x": (_int, [_vp, _i64, _i64, _vp, _vp, _vp, _vp, _vp, _vp, _sz, _vp]),
    "tqfx4_expert_ffn_workspace_bytes": (_sz, [_i64, _i64]),
    "tqfx4_expert_ffn_launches": (_int, [_i64, _i64]),
    "tqfx4_expert_ffn": (_int, [_vp, _vp, _vp, _i64, _i64, _vp, _vp, _vp, _sz, _vp]),
    "tqfx4_expert_ffn_traced": (_int, [_vp, _vp, _vp, _i64, _i64, _vp, _vp, _vp, _sz, _vp, _vp]),
    "tqfx4_moe_workspace_bytes": (_sz, [C.POINTER(CExperts), C.POINTER(CRouter), _i64, _int]),
    "tqfx4_moe_ffn": (_int, [C.POINTER(CExperts), C.POINTER(CRouter), _vp, _vp, _vp, _vp, _vp, _sz, _vp]),
    "tqfx4_validate_blocks": (_int, [_vp, _i64, _i64, _vp, _sz, _vp]),
    "tqfx4_moe_grouped_host": (_int, [C.POINTER(CExperts), C.POINTER(CRouter), _vp, _i64, _vp, _vp, _vp, _int,
                                      _vp, _sz, _vp]),
    "tqfx4_moe_grouped_host_workspace_bytes": (_sz, [C.POINTER(CExperts), C.POINTER(CRouter), _i64, _int]),
    "tqfx4_moe_ffn_host": (_int, [C.POINTER(CExperts), C.POINTER(CRouter), _vp, _vp, _vp, _vp, _vp, _sz, _vp]),
    "tqfx4_gemv_x_host": (_int, [_vp, _i64, _i64, _vp, _vp, _vp, _sz, _vp]),
    "tqfx4_gemv_x_host_workspace_bytes": (_sz, [_i64, _i64]),
    "tqfx4_expert_ffn_host": (_int, [_vp, _vp, _vp, _i64, _i64, _vp, _vp, _vp, _sz, _vp]),
    "tqfx4_expert_ffn_host_workspace_bytes": (_sz, [_i64, _i64]),
    "tqfx4_moe_ffn_host_workspace_bytes": (_sz, [C.POINTER(CExperts), C.POINTER(CRouter)]),
    "tqfx4_moe_ffn_mxfp4": (_int, [C.POINTER(CExperts), C.POINTER(CRouter), _vp, _vp, _vp, _vp, _vp, _sz, _vp]),
    "tqfx4_moe_ffn_mxfp4_traced": (_int, [C.POINTER(CExperts), C.POINTER(CRouter), _vp, _vp, _vp, _vp, _vp, _sz,
                                          _vp, C.POINTER(_vp)]),
    "tqfx4_moe_grouped": (_int, [C.POINTER(CExperts), C.POINTER(CRouter), _vp, _i64, _vp, _vp, _vp, _int,
                                 _vp, _sz, _vp]),
    "tqfx4_moe_stage_count": (_int, [_int, _int]),
    "tqfx4_moe_stage_name": (C.c_char_p, [_int, _int, _int]),
    "tqfx4_moe_ffn_traced": (_int, [C.POINTER(CExperts), C.POINTER(CRouter), _vp, _vp, _vp, _vp, _vp, _sz,
                                    _vp, C.POINTER(_vp)]),
    "tqfx4_moe_grouped_traced": (_int, [C.POINTER(CExperts), C.POINTER(CRouter), _vp, _i64, _vp, _vp, _vp,
                                        _int, _vp, _sz, _vp, C.POINTER(_vp)]),
    "tqfx4_moe_workspace_views": (_int, [C.POINTER(CExperts), C.POINTER(CRouter), _i64, _int, _int,
                                         C.POINTER(CMoeViews)]),
    "tqfx4_moe_ffn_noalloc": (_int, [C.POINTER(CExperts), C.POINTER(CRouter), _vp, _vp, _vp, _vp, _vp]),
    "tqfx4_free_bytes": (_i64, [_i64, _i64]),
    "tqfx4_pack_free": (_int, [_vp, _vp, _vp, _vp, _i64, _i64, _vp, _vp, _sz, _vp]),
    "tqfx4_gemv_free": (_int, [_vp, _i64, _i64, _vp, _vp, _vp, _vp, _vp, _vp, _vp, _sz, _vp]),
    "tqfx4_mxfp4_bytes": (_i64, [_i64, _i64]),
    "tqfx4_gemv_mxfp4": (_int, [_vp, _i64, _i64, _vp, _vp, _vp, _vp, _vp, _sz, _vp]),
    "tqfx4_moe_route": (_int, [C.POINTER(CExperts), C.POINTER(CRouter), _vp, _vp, _vp, _vp, _sz, _vp]),
    "tqfx4_moe_experts": (_int, [C.POINTER(CExperts), C.POINTER(CRouter), _vp, _vp, _vp, _sz, _vp]),
    "tqfx4_check": (_int, [_vp, _vp]),
    "tqfx4_selftest_wait_timeout": (_int, [_vp, _sz, _vp]),
    "tqfx4_last_error": (C.c_char_p, []),
    "tqfx4_status_string": (C.c_char_p, [_int]),
}

_lib = None


def load(path: str):
    """A library of this ABI at `path`, with every declared signature set."""
    if not os.path.exists(path):
        raise RuntimeError("%s is not built; run __graft_entry__.build()" % path)
    L = C.CDLL(path)
    for name, (res, args) in _SIGS.items():
        f = getattr(L, name)  # a missing export is a build error: raise here
        f.restype = res
        f.argtypes = args
    return L


def lib():
    """Load libtqfx4.so (built in-tree by __graft_entry__.build())."""
    global _lib
    if _lib is None:
        _lib = load(LIB_PATH)
    return _lib


def _p(t):
    if t is None:
        return None
    if isinstance(t, int):
        return t
    return t.data_ptr()


def _s(stream):
    if stream is None:
        return torch.cuda.current_stream().cuda_stream
    if isinstance(stream, int):
        return stream
    return stream.cuda_stream


def _check(rc, fn):
    if rc != 0:
        msg = lib().tqfx4_last_error().decode(errors="replace")
        raise TqfxError(rc, fn, msg)


def _nbytes(t):
    return 0 if t is None else t.numel() * t.element_size()


# ---------------------------------------------------------------- format

def tqfx4_matrix_bytes(n: int, k: int) -> int:
    return int(lib().tqfx4_matrix_bytes(n, k))


def tqfx4_basic_workspace_bytes() -> int:
    return int(lib().tqfx4_basic_workspace_bytes())


def tqfx4_pack(src, a, t2, scales_f16, n, k, blocks, ws, stream=None):
    _check(lib().tqfx4_pack(src, _p(a), _p(t2), _p(scales_f16), n, k, _p(blocks), _p(ws), _nbytes(ws),
                            _s(stream)), "tqfx4_pack")


def tqfx4_quantize_act(x, m, k, q, da, bsum, ws, stream=None):
    _check(lib().tqfx4_quantize_act(_p(x), m, k, _p(q), _p(da), _p(bsum), _p(ws), _nbytes(ws), _s(stream)),
           "tqfx4_quantize_act")


def tqfx4_gemv(blocks, n, k, q, da, bsum, y, block_sums, ws, stream=None):
    _check(lib().tqfx4_gemv(_p(blocks), n, k, _p(q), _p(da), _p(bsum), _p(y), _p(block_sums), _p(ws),
                            _nbytes(ws), _s(stream)), "tqfx4_gemv")


def tqfx4_expert_ffn_workspace_bytes(hidden, inter):
    return lib().tqfx4_expert_ffn_workspace_bytes(hidden, inter)


def tqfx4_expert_ffn_launches(hidden, inter):
    return int(lib().tqfx4_expert_ffn_launches(hidden, inter))


def tqfx4_expert_ffn(gate, up, down, hidden, inter, x, out, ws, stream=None, events=None):
    if events is None:
        rc = lib().tqfx4_expert_ffn(_p(gate), _p(up), _p(down), hidden, inter, _p(x), _p(out), _p(ws), _nbytes(ws),
                                    _s(stream))
    else:
        arr = (_vp * len(events))(*[e.cuda_event if hasattr(e, "cuda_event") else e for e in events])
        rc = lib().tqfx4_expert_ffn_traced(_p(gate), _p(up), _p(down), hidden, inter, _p(x), _p(out), _p(ws),
                                           _nbytes(ws), _s(stream), arr)
    _check(rc, "tqfx4_expert_ffn")


def tqfx4_gemv_x(blocks, n, k, x, y, q, da, bsum, ws, stream=None):
    _check(lib().tqfx4_gemv_x(_p(blocks), n, k, _p(x), _p(y), _p(q), _p(da), _p(bsum), _p(ws), _nbytes(ws),
                              _s(stream)), "tqfx4_gemv_x")


# ---------------------------------------------------------------- MoE

def c_experts(gate, up, down, n_experts, hidden, inter) -> CExperts:
    return CExperts(_p(gate), _p(up), _p(down), n_experts, hidden, inter)


def c_router(weight, bias, top_k) -> CRouter:
    return CRouter(_p(weight), _p(bias), top_k)


def tqfx4_moe_workspace_bytes(ex: CExperts, rt: CRouter, tokens: int, path: int = 0) -> int:
    return int(lib().tqfx4_moe_workspace_bytes(C.byref(ex), C.byref(rt), tokens, path))


def tqfx4_moe_ffn(ex, rt, x, out, sel_idx, sel_w, ws, stream=None, events=None):
    if events is None:
        rc = lib().tqfx4_moe_ffn(C.byref(ex), C.byref(rt), _p(x), _p(out), _p(sel_idx), _p(sel_w), _p(ws),
                                 _nbytes(ws), _s(stream))
    else:
        arr = (_vp * len(events))(*[e.cuda_event if hasattr(e, "cuda_event") else e for e in events])
        rc = lib().tqfx4_moe_ffn_traced(C.byref(ex), C.byref(rt), _p(x), _p(out), _p(sel_idx), _p(sel_w),
                                        _p(ws), _nbytes(ws), _s(stream), arr)
    _check(rc, "tqfx4_moe_ffn")


def tqfx4_validate_blocks(blocks, n, k, ws, stream=None):
    """Checks the format of an n x k matrix (nibbles 0..8, finite scales); a
    violation shows in tqfx4_check(ws) as TQFX4_EDATA."""
    _check(lib().tqfx4_validate_blocks(_p(blocks), n, k, _p(ws), _nbytes(ws), _s(stream)), "tqfx4_validate_blocks")


def tqfx4_moe_grouped_host_workspace_bytes(ex: CExperts, rt: CRouter, tokens: int, path: int = 0) -> int:
    return int(lib().tqfx4_moe_grouped_host_workspace_bytes(C.byref(ex), C.byref(rt), tokens, path))


def tqfx4_moe_grouped_host(ex, rt, X, T, OUT, sel_idx, sel_w, path, ws, stream=None):
    """X, OUT, sel_idx, sel_w: CPU tensors (page-locked: used in place);
    sel_idx and sel_w may be None. Complete once `stream` has passed the call."""
    _check(lib().tqfx4_moe_grouped_host(C.byref(ex), C.byref(rt), _p(X), T, _p(OUT), _p(sel_idx), _p(sel_w), path,
                                        _p(ws), _nbytes(ws), _s(stream)), "tqfx4_moe_grouped_host")


def tqfx4_gemv_x_host_workspace_bytes(n: int, k: int) -> int:
    return int(lib().tqfx4_gemv_x_host_workspace_bytes(n, k))


def tqfx4_gemv_x_host(blocks, n, k, x, y, ws, stream=None):
    """x, y: CPU tensors (page-locked: used in place); y is complete once
    `stream` has passed the call."""
    _check(lib().tqfx4_gemv_x_host(_p(blocks), n, k, _p(x), _p(y), _p(ws), _nbytes(ws), _s(stream)),
           "tqfx4_gemv_x_host")


def tqfx4_expert_ffn_host_workspace_bytes(hidden: int, inter: int) -> int:
    return int(lib().tqfx4_expert_ffn_host_workspace_bytes(hidden, inter))


def tqfx4_expert_ffn_host(gate, up, down, hidden, inter, x, out, ws, stream=None):
    """x, out: CPU tensors (page-locked: used in place); out is complete once
    `stream` has passed the call."""
    _check(lib().tqfx4_expert_ffn_host(_p(gate), _p(up), _p(down), hidden, inter, _p(x), _p(out), _p(ws),
                                       _nbytes(ws), _s(stream)), "tqfx4_expert_ffn_host")


def tqfx4_moe_ffn_host_workspace_bytes(ex: CExperts, rt: CRouter) -> int:
    return int(lib().tqfx4_moe_ffn_host_workspace_bytes(C.byref(ex), C.byref(rt)))


def tqfx4_moe_ffn_host(ex, rt, x, out, sel_idx, sel_w, ws, stream=None):
    """x, out, sel_idx, sel_w: CPU tensors (page-locked for asynchronous copies);
    sel_idx and sel_w may be None. The outputs are complete once `stream` has
    passed the call."""
    _check(lib().tqfx4_moe_ffn_host(C.byref(ex), C.byref(rt), _p(x), _p(out), _p(sel_idx), _p(sel_w), _p(ws),
                                    _nbytes(ws), _s(stream)), "tqfx4_moe_ffn_host")


def tqfx4_moe_ffn_mxfp4(ex, rt, x, out, sel_idx, sel_w, ws, stream=None, events=None):
    if events is None:
        rc = lib().tqfx4_moe_ffn_mxfp4(C.byref(ex), C.byref(rt), _p(x), _p(out), _p(sel_idx), _p(sel_w), _p(ws),
                                       _nbytes(ws), _s(stream))
    else:
        arr = (_vp * len(events))(*[e.cuda_event if hasattr(e, "cuda_event") else e for e in events])
        rc = lib().tqfx4_moe_ffn_mxfp4_traced(C.byref(ex), C.byref(rt), _p(x), _p(out), _p(sel_idx), _p(sel_w),
                                              _p(ws), _nbytes(ws), _s(stream), arr)
    _check(rc, "tqfx4_moe_ffn_mxfp4")


def tqfx4_moe_ffn_noalloc(ex, rt, x, out, sel_idx, sel_w, stream=None):
    """tqfx4_moe_ffn on the library's own scratch (for callers that cannot
    allocate device memory; see include/tqfx4.h)."""
    _check(lib().tqfx4_moe_ffn_noalloc(C.byref(ex), C.byref(rt), _p(x), _p(out), _p(sel_idx), _p(sel_w),
                                       _s(stream)), "tqfx4_moe_ffn_noalloc")


def tqfx4_free_bytes(n: int, k: int) -> int:
    return int(lib().tqfx4_free_bytes(n, k))


def tqfx4_pack_free(t1, t2, a1, a2, n, k, blocks, ws, stream=None):
    _check(lib().tqfx4_pack_free(_p(t1), _p(t2), _p(a1), _p(a2), n, k, _p(blocks), _p(ws), _nbytes(ws),
                                 _s(stream)), "tqfx4_pack_free")


def tqfx4_gemv_free(blocks, n, k, q, da, bsum, y, S1, S2, ws, stream=None):
    _check(lib().tqfx4_gemv_free(_p(blocks), n, k, _p(q), _p(da), _p(bsum), _p(y), _p(S1), _p(S2), _p(ws),
                                 _nbytes(ws), _s(stream)), "tqfx4_gemv_free")


def tqfx4_mxfp4_bytes(n: int, k: int) -> int:
    return int(lib().tqfx4_mxfp4_bytes(n, k))


def tqfx4_gemv_mxfp4(blocks, n, k, q, da, y, block_sums, ws, stream=None):
    _check(lib().tqfx4_gemv_mxfp4(_p(blocks), n, k, _p(q), _p(da), _p(y), _p(block_sums), _p(ws), _nbytes(ws),
                                  _s(stream)), "tqfx4_gemv_mxfp4")


def tqfx4_moe_route(ex, rt, x, sel_idx, sel_w, ws, stream=None):
    _check(lib().tqfx4_moe_route(C.byref(ex), C.byref(rt), _p(x), _p(sel_idx), _p(sel_w), _p(ws), _nbytes(ws),
                                 _s(stream)), "tqfx4_moe_route")


def tqfx4_moe_experts(ex, rt, ptrs, out, ws, stream=None):
    """ptrs: a device int64 tensor of 3 x top_k block addresses (gate, up,
    down of the selected experts in rank order)."""
    _check(lib().tqfx4_moe_experts(C.byref(ex), C.byref(rt), _p(ptrs), _p(out), _p(ws), _nbytes(ws), _s(stream)),
           "tqfx4_moe_experts")


def tqfx4_moe_grouped(ex, rt, X, T, OUT, sel_idx, sel_w, path, ws, stream=None, events=None):
    if events is None:
        rc = lib().tqfx4_moe_grouped(C.byref(ex), C.byref(rt), _p(X), T, _p(OUT), _p(sel_idx), _p(sel_w),
                                     path, _p(ws), _nbytes(ws), _s(stream))
    else:
        arr = (_vp * len(events))(*[e.cuda_event if hasattr(e, "cuda_event") else e for e in events])
        rc = lib().tqfx4_moe_grouped_traced(C.byref(ex), C.byref(rt), _p(X), T, _p(OUT), _p(sel_idx),
                                            _p(sel_w), path, _p(ws), _nbytes(ws), _s(stream), arr)
    _check(rc, "tqfx4_moe_grouped")


def tqfx4_moe_stage_count(grouped: int, path: int) -> int:
    return int(lib().tqfx4_moe_stage_count(grouped, path))


def tqfx4_moe_stage_name(grouped: int, path: int, stage: int) -> str:
    return lib().tqfx4_moe_stage_name(grouped, path, stage).decode()


def tqfx4_moe_workspace_views(ex, rt, tokens, grouped, path) -> dict:
    v = CMoeViews()
    _check(lib().tqfx4_moe_workspace_views(C.byref(ex), C.byref(rt), tokens, grouped, path, C.byref(v)),
           "tqfx4_moe_workspace_views")
    return {name: getattr(v, name) for name, _ in CMoeViews._fields_}


def tqfx4_check(ws, stream=None):
    _check(lib().tqfx4_check(_p(ws), _s(stream)), "tqfx4_check")


def tqfx4_selftest_wait_timeout(ws, stream=None):
    _check(lib().tqfx4_selftest_wait_timeout(_p(ws), _nbytes(ws), _s(stream)), "tqfx4_selftest_wait_timeout")


def tqfx4_last_error() -> str:
    return lib().tqfx4_last_error().decode(errors="replace")
