"""The C-ABI library without a GPU: it loads, exports every function that
include/tqfx4.h declares, and its host-side logic (sizes, workspace layout,
stage names, argument validation) answers before any device work.

No call here reaches a kernel: every compute call is made with arguments the
library must reject on the host, and the test checks the status it returns.
"""
import ctypes as C
import os
import re

import pytest

import oracle
from paper_2608_08910_gb300 import binding as B

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "tqfx4.h")


@pytest.fixture(scope="module")
def lib():
    if not os.path.exists(B.LIB_PATH):
        from paper_2608_08910_gb300 import build
        build.build()
    return B.lib()


def declared_functions():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    text = re.sub(r"//[^\n]*", "", text)
    names = set(re.findall(r"\b(tqfx4_[a-z0-9_]+)\s*\(", text))
    return sorted(names)


def test_header_declares_the_calls_of_the_path():
    names = declared_functions()
    for fn in ("tqfx4_pack", "tqfx4_quantize_act", "tqfx4_gemv", "tqfx4_moe_ffn", "tqfx4_moe_grouped"):
        assert fn in names


def test_library_exports_every_declared_function(lib):
    raw = C.CDLL(B.LIB_PATH)
    missing = [n for n in declared_functions() if not hasattr(raw, n)]
    assert not missing, missing
    # and the binding declares a signature for each of them
    assert set(declared_functions()) <= set(B._SIGS)


def test_matrix_bytes_match_the_format(lib):
    for n, k in [(4, 256), (1024, 1024), (2048, 4096), (4096, 2048), (8, 512)]:
        assert lib.tqfx4_matrix_bytes(n, k) == oracle.matrix_bytes(n, k) == (n // 4) * (k // 256) * 520
    assert lib.tqfx4_matrix_bytes(6, 256) < 0  # rows not a multiple of 4
    assert lib.tqfx4_matrix_bytes(4, 100) < 0  # k not a multiple of 256


def test_debug_library_builds_and_exports_the_same_functions():
    # the TQFX4_DEBUG variant (format validation in the entry points, index
    # checks in the kernels) compiles for sm_103a and carries the whole ABI
    from paper_2608_08910_gb300 import build
    path = build.build(debug=True)
    raw = C.CDLL(path)
    missing = [n for n in declared_functions() if not hasattr(raw, n)]
    assert not missing, missing


def test_status_strings(lib):
    for code, name in B.STATUS_NAMES.items():
        assert lib.tqfx4_status_string(code).decode() == name


def shapes(E=256, H=4096, I=2048, k=8):
    return B.CExperts(None, None, None, E, H, I), B.CRouter(None, None, k)


def test_moe_workspace_layout(lib):
    ex, rt = shapes()
    for T, grouped in [(1, 0), (64, 1), (2048, 1)]:
        v = B.CMoeViews()
        assert lib.tqfx4_moe_workspace_views(C.byref(ex), C.byref(rt), T, grouped, 0, C.byref(v)) == 0
        total = lib.tqfx4_moe_workspace_bytes(C.byref(ex), C.byref(rt), T, 0)
        P = T * 8
        spans = {"logits": 4 * T * 256, "qx": T * 4096, "g": 4 * P * 2048, "u": 4 * P * 2048,
                 "h": 4 * P * 2048, "qh": P * 2048, "o": 4 * P * 4096}
        if grouped:
            spans.update(counts=4 * 256, pair_token=4 * P, pair_of=4 * P)
        ranges = sorted((getattr(v, n), getattr(v, n) + s) for n, s in spans.items())
        assert ranges[0][0] >= B.TQFX4_STATUS_BYTES  # the status word comes first
        for (a0, a1), (b0, b1) in zip(ranges, ranges[1:]):
            assert a1 <= b0  # disjoint
        assert ranges[-1][1] <= total
        assert all(getattr(v, n) % 256 == 0 for n in spans)


def test_stage_names(lib):
    assert lib.tqfx4_moe_stage_count(0, 0) == 3
    assert [lib.tqfx4_moe_stage_name(0, 0, s).decode() for s in range(3)] == ["router", "gate_up", "down"]
    n = lib.tqfx4_moe_stage_count(1, 0)
    names = [lib.tqfx4_moe_stage_name(1, 0, s).decode() for s in range(n)]
    assert names[0] == "router" and "gate_up" in names and "down" in names and names[-1] == "combine"
    assert lib.tqfx4_moe_stage_name(1, 0, n).decode() == ""


def test_host_validation_rejects_bad_arguments(lib):
    # shapes first, then pointers and workspace: all decided on the host
    assert lib.tqfx4_gemv(None, 1023, 1024, None, None, None, None, None, None, 0, None) == 2
    assert lib.tqfx4_gemv(None, 1024, 1000, None, None, None, None, None, None, 0, None) == 2
    assert lib.tqfx4_gemv(None, 1024, 1024, None, None, None, None, None, None, 0, None) == 1
    assert lib.tqfx4_quantize_act(None, 1, 100, None, None, None, None, 0, None) == 2
    # the expert FFN's workspace: the one-expert, top-1 decode layout (at most
    # the MoE call's, which also covers the grouped layout); 0 for bad shapes
    ex1, rt1 = shapes(E=1, k=1)
    n1 = lib.tqfx4_expert_ffn_workspace_bytes(4096, 2048)
    assert 0 < n1 <= lib.tqfx4_moe_workspace_bytes(C.byref(ex1), C.byref(rt1), 1, 0)
    assert lib.tqfx4_expert_ffn_workspace_bytes(4000, 2048) == 0
    assert lib.tqfx4_expert_ffn_workspace_bytes(4096, 0) == 0
    # one cooperative launch where the expert fits on chip with even block
    # counts, else two; 0 for bad shapes
    assert lib.tqfx4_expert_ffn_launches(4096, 2048) == 1
    assert lib.tqfx4_expert_ffn_launches(768, 1280) == 2
    assert lib.tqfx4_expert_ffn_launches(4096, 8192) == 2
    assert lib.tqfx4_expert_ffn_launches(4000, 2048) == 0
    # the one-launch GEMV takes the chunked pass only: k a multiple of 512
    assert lib.tqfx4_gemv_x(None, 1024, 256, None, None, None, None, None, None, 0, None) == 2
    assert lib.tqfx4_gemv_x(None, 1024, 1280, None, None, None, None, None, None, 0, None) == 2
    assert lib.tqfx4_gemv_x(None, 1024, 1024, None, None, None, None, None, None, 0, None) == 1
    # the host-buffer MoE call: staging after the decode layout; NULL host
    # buffers and bad shapes are refused before any copy
    exh, rth = shapes()
    nh = lib.tqfx4_moe_ffn_host_workspace_bytes(C.byref(exh), C.byref(rth))
    assert nh >= 2 * 4 * 4096 + 2 * 4 * 8 and nh % 256 == 0
    assert lib.tqfx4_moe_ffn_host_workspace_bytes(C.byref(ex_bad_h := shapes(H=4000)[0]), C.byref(rth)) == 0
    assert lib.tqfx4_moe_ffn_host(C.byref(exh), C.byref(rth), None, None, None, None, None, 0, None) == 1
    assert lib.tqfx4_moe_ffn_host(C.byref(ex_bad_h), C.byref(rth), None, None, None, None, None, 0, None) == 2
    # the host-buffer GEMV and expert FFN: status word and staging; shape and
    # NULL errors before any copy
    assert lib.tqfx4_gemv_x_host_workspace_bytes(1024, 1024) >= B.TQFX4_STATUS_BYTES + 8 * 1024
    assert lib.tqfx4_gemv_x_host_workspace_bytes(1024, 256) == 0
    assert lib.tqfx4_gemv_x_host(None, 1024, 256, None, None, None, 0, None) == 2
    assert lib.tqfx4_gemv_x_host(None, 1024, 1024, None, None, None, 0, None) == 1  # workspace first
    ne = lib.tqfx4_expert_ffn_host_workspace_bytes(4096, 2048)
    assert ne >= lib.tqfx4_expert_ffn_workspace_bytes(4096, 2048) + 2 * 4 * 4096
    assert lib.tqfx4_expert_ffn_host_workspace_bytes(4000, 2048) == 0
    assert lib.tqfx4_expert_ffn_host(None, None, None, 4000, 2048, None, None, None, 0, None) == 2
    assert lib.tqfx4_expert_ffn_host(None, None, None, 4096, 2048, None, None, None, 0, None) == 1
    # the host-buffer grouped call
    exg, rtg = shapes()
    ng = lib.tqfx4_moe_grouped_host_workspace_bytes(C.byref(exg), C.byref(rtg), 64, 0)
    assert ng >= lib.tqfx4_moe_workspace_bytes(C.byref(exg), C.byref(rtg), 64, 0) + 2 * 64 * 4096 * 4
    assert lib.tqfx4_moe_grouped_host_workspace_bytes(C.byref(exg), C.byref(rtg), 0, 0) == 0
    assert lib.tqfx4_moe_grouped_host(C.byref(exg), C.byref(rtg), None, 0, None, None, None, 0, None, 0,
                                      None) == 0  # no tokens: nothing to do
    assert lib.tqfx4_moe_grouped_host(C.byref(exg), C.byref(rtg), None, -1, None, None, None, 0, None, 0,
                                      None) == 1
    # the format check: shapes, then the workspace, then NULL blocks
    assert lib.tqfx4_validate_blocks(None, 6, 256, None, 0, None) == 2
    assert lib.tqfx4_validate_blocks(None, 4, 256, None, 0, None) == 1
    assert lib.tqfx4_pack(7, None, None, None, 4, 256, None, None, 0, None) == 1  # unknown source kind
    ex, rt = shapes()
    assert lib.tqfx4_moe_ffn(C.byref(ex), C.byref(rt), None, None, None, None, None, 0, None) == 1
    ex_bad, rt_bad = shapes(H=4000)
    assert lib.tqfx4_moe_workspace_bytes(C.byref(ex_bad), C.byref(rt), 1, 0) == 0
    _, rt_k = shapes(k=300)
    assert lib.tqfx4_moe_workspace_bytes(C.byref(ex), C.byref(rt_k), 1, 0) == 0
    ex_odd, _ = shapes(H=768)  # 3 blocks per row: valid for decode, not for the grouped path
    assert lib.tqfx4_moe_grouped(C.byref(ex_odd), C.byref(rt), None, 2, None, None, None, 0, None, 0,
                                 None) == 2
    assert lib.tqfx4_moe_grouped(C.byref(ex), C.byref(rt), None, 2, None, None, None, 9, None, 0, None) == 1
    assert b"path" in lib.tqfx4_last_error()
