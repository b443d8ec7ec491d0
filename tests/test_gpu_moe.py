"""GPU parity of tqfx4_moe_ffn (one token through a routed-expert MoE layer)
against the CPU oracle, through the C ABI.

Checked per token: the routing decision (expert ids bit-exact unless the
oracle puts two candidates within the error bound of the two logit
evaluations, in
which case either order is valid), the quantized hidden state, each selected
expert's g, u, h, re-quantized h and down output (bit-exact: the kernels use
the oracle's float schedule and the same specified binary32 SwiGLU), and the
combined output within 1e-4 relative.
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2608_08910_gb300 import binding as B
from paper_2608_08910_gb300 import inputs
from paper_2608_08910_gb300.moe import MoeLayer
from tests.parity import FP32_TOL, check_selection, oracle_experts, rel_err, selection_tolerance

pytestmark = pytest.mark.gpu
DEV = "cuda"


def run_and_check(layer, seed, X, zipf_bias=None, check_stages=True):
    H, I, E, k = layer.hidden, layer.inter, layer.n_experts, layer.top_k
    ws = layer.workspace(1)
    Wr = layer.router_w.cpu().numpy()
    bias = None if layer.router_b is None else layer.router_b.cpu().numpy()
    worst = 0.0
    for t in range(X.shape[0]):
        x = X[t]
        out, sel, selw = layer.ffn(x.to(DEV), ws)
        B.tqfx4_check(ws)
        out, sel, selw = out.cpu().numpy(), sel.cpu().numpy(), selw.cpu().numpy()
        logits, r_idx, r_w = oracle.router(Wr, bias, x.numpy(), k)
        tol = selection_tolerance(Wr, x.numpy(), bias)
        hi = layer.view(ws, "logits", torch.float32, (E,)).cpu().numpy().astype(np.float64)
        lo = layer.view(ws, "logits_lo", torch.float32, (E,)).cpu().numpy().astype(np.float64)
        assert np.all(np.abs((hi + lo) - logits) <= tol)
        assert np.all(np.abs(lo) <= np.spacing(np.abs(hi).astype(np.float32)))  # normalized pairs
        ties = check_selection(sel, logits, tol, k)
        ex = oracle_experts(seed, np.union1d(sel, r_idx), H, I)
        ref, _, _ = oracle.moe_tokens(ex, E, H, I, Wr, bias, k, x.numpy())
        if ties == 0:
            assert np.array_equal(sel, r_idx)
            assert np.allclose(selw, r_w, rtol=1.2e-7, atol=0)  # fp64 softmax, one rounding
            e_ = rel_err(out, ref[0])
            assert e_ <= FP32_TOL, e_
            worst = max(worst, e_)
        if check_stages:
            rq, rdx, rbx = oracle.quantize_act(x.numpy())
            assert np.array_equal(layer.view(ws, "qx", torch.int8, (H,)).cpu().numpy(), rq)
            g = layer.view(ws, "g", torch.float32, (k, I)).cpu().numpy()
            u = layer.view(ws, "u", torch.float32, (k, I)).cpu().numpy()
            h = layer.view(ws, "h", torch.float32, (k, I)).cpu().numpy()
            qh = layer.view(ws, "qh", torch.int8, (k, I)).cpu().numpy()
            o = layer.view(ws, "o", torch.float32, (k, H)).cpu().numpy()
            for j, e in enumerate(sel):
                ro, dbg = oracle.expert_ffn(*ex[int(e)], H, I, x.numpy())
                assert np.array_equal(g[j], dbg["g"]) and np.array_equal(u[j], dbg["u"])
                assert np.array_equal(h[j].view(np.uint32), dbg["h"].view(np.uint32))
                assert np.array_equal(qh[j], dbg["qh"])
                assert np.array_equal(o[j].view(np.uint32), ro.view(np.uint32))
            # the combine in rank order with the kernel's own weights is exact
            acc = np.zeros(H, np.float32)
            for j in range(k):
                acc = (acc + np.float32(selw[j]) * o[j]).astype(np.float32)
            assert np.array_equal(acc.view(np.uint32), out.view(np.uint32))
    return worst


@pytest.mark.parametrize("E,H,I,k,zipf", [(16, 512, 768, 4, 0.0), (8, 256, 256, 8, 0.0), (32, 1024, 512, 6, 1.1),
                                          (1, 256, 512, 1, 0.0), (64, 2048, 1280, 8, 0.0),
                                          (300, 256, 256, 16, 0.5),    # 16 keys per lane in the top-k, k at its maximum
                                          (1024, 256, 256, 12, 1.1)])  # 32 keys per lane, the largest expert count
def test_moe_ffn_small_shapes(E, H, I, k, zipf):
    seed = E * 7 + H + I
    layer = MoeLayer.synthetic(seed, E, H, I, k, zipf, DEV)
    X = inputs.hidden_states(seed, 3, H)
    run_and_check(layer, seed, X)


# hidden and intermediate sizes from 512 to 8192 (rows of 2 to 32 blocks),
# fewer and more experts than SMs, top-k up to 16 and a top-k of 7 (row
# ranges that do not divide evenly)
@pytest.mark.parametrize("E,H,I,k,zipf", [(64, 1024, 2048, 8, 0.0), (16, 2048, 512, 4, 1.1),
                                          (1024, 512, 1024, 16, 0.5), (12, 4096, 4096, 7, 0.0),
                                          (8, 8192, 1024, 3, 0.0), (8, 1024, 8192, 2, 0.0)])
def test_moe_ffn_more_shapes(E, H, I, k, zipf):
    seed = E * 5 + H + 3 * I
    layer = MoeLayer.synthetic(seed, E, H, I, k, zipf, DEV)
    X = inputs.hidden_states(seed, 3, H)
    run_and_check(layer, seed, X)


def test_one_expert_ffn_full_size():
    # the batch-1 SwiGLU expert, gate/up 4096->2048 and down 2048->4096
    layer = MoeLayer.synthetic(1, 1, 4096, 2048, 1, 0.0, DEV)
    X = inputs.hidden_states(1, 2, 4096)
    ws = layer.workspace(1)
    ex = oracle_experts(1, [0], 4096, 2048)
    g, u, d = layer.expert_blocks(0)
    for e_, blk in zip(ex[0], (g, u, d)):
        assert np.array_equal(blk.cpu().numpy(), e_)
    for t in range(2):
        out, sel, selw = layer.ffn(X[t].to(DEV), ws)
        B.tqfx4_check(ws)
        ref, _ = oracle.expert_ffn(*ex[0], 4096, 2048, X[t].numpy())
        assert sel.item() == 0 and selw.item() == 1.0
        assert np.array_equal(out.cpu().numpy().view(np.uint32), ref.view(np.uint32))


@pytest.fixture(scope="module")
def full_layer():
    return MoeLayer.synthetic(0, 256, 4096, 2048, 8, 0.0, DEV)


def test_moe_decode_full_size(full_layer):
    # 256 experts, hidden 4096, expert-intermediate 2048, top-8: sampled tokens
    X = inputs.hidden_states(0, 3, 4096)
    run_and_check(full_layer, 0, X)


def test_moe_decode_is_deterministic(full_layer):
    x = inputs.hidden_states(5, 1, 4096)[0].to(DEV)
    ws = full_layer.workspace(1)
    a = [t.clone() for t in full_layer.ffn(x, ws)]
    b = full_layer.ffn(x, ws)
    for p, q in zip(a, b):
        assert torch.equal(p, q)


def test_moe_decode_many_calls_in_a_row(full_layer):
    # the cross-CTA counters return to zero after every call: 50 calls on one
    # workspace, alternating two tokens, each equal to the first call's result
    X = inputs.hidden_states(6, 2, 4096).to(DEV)
    ws = full_layer.workspace(1)
    ref = [[t.clone() for t in full_layer.ffn(X[i], ws)] for i in range(2)]
    outs = []
    for c in range(50):
        outs.append(full_layer.ffn(X[c % 2], ws)[0].clone())
    B.tqfx4_check(ws)
    for c, o in enumerate(outs):
        assert torch.equal(o, ref[c % 2][0])


def host_buffer(v, kind):
    """v in host memory: page-locked, pageable, or page-locked 4 bytes off
    16-byte alignment."""
    if kind == "pinned":
        return v.clone().pin_memory()
    if kind == "pageable":
        return v.clone()
    buf = torch.empty(v.numel() + 1, dtype=v.dtype).pin_memory()
    buf[1:] = v
    return buf[1:]


@pytest.mark.parametrize("kind", ["pinned", "pageable", "pinned_unaligned"])
def test_moe_ffn_host_equals_the_device_call(full_layer, kind):
    # the host-buffer entry point brings x in and out, sel_idx and sel_w back
    # on the stream (page-locked buffers in place, the others through staging
    # copies): the same bits as the device call, token after token on one
    # workspace
    X = inputs.hidden_states(7, 4, 4096)
    ws = full_layer.workspace(1)
    wsh = full_layer.host_workspace()
    stream = torch.cuda.current_stream()
    for t in range(X.shape[0]):
        ref = [v.cpu() for v in full_layer.ffn(X[t].to(DEV), ws)]
        xh = host_buffer(X[t], kind)
        outh = host_buffer(torch.zeros(4096), kind)
        selh = host_buffer(torch.zeros(8, dtype=torch.int32), kind)
        wh = host_buffer(torch.zeros(8), kind)
        full_layer.ffn_host(xh, wsh, outh, selh, wh, stream=stream)
        stream.synchronize()
        B.tqfx4_check(wsh)
        assert torch.equal(outh.view(torch.int32), ref[0].view(torch.int32)), t
        assert torch.equal(selh, ref[1]), t
        assert torch.equal(wh.view(torch.int32), ref[2].view(torch.int32)), t
    # the selection outputs are optional
    outh = torch.empty(4096).pin_memory()
    full_layer.ffn_host(X[0].clone().pin_memory(), wsh, outh, None, None, stream=stream)
    stream.synchronize()
    ref0 = full_layer.ffn(X[0].to(DEV), ws)[0].cpu()
    assert torch.equal(outh.view(torch.int32), ref0.view(torch.int32))


@pytest.mark.parametrize("kind", ["pinned", "pageable", "pinned_unaligned"])
def test_expert_ffn_host_equals_the_device_call(kind):
    # x and out in host memory (page-locked: x read by a small kernel, out
    # written in place by the down kernel; others through staging copies):
    # out bit-identical to expert_ffn's, 4 tokens on one workspace
    layer = MoeLayer.synthetic(31, 1, 4096, 2048, 1, 0.0, DEV)
    ws = layer.expert_workspace()
    wsh = layer.expert_host_workspace()
    stream = torch.cuda.current_stream()
    X = inputs.hidden_states(31, 4, 4096)
    for t in range(X.shape[0]):
        ref = layer.expert_ffn(0, X[t].to(DEV), ws).cpu()
        xh, oh = host_buffer(X[t], kind), host_buffer(torch.zeros(4096), kind)
        layer.expert_ffn_host(0, xh, wsh, oh, stream=stream)
        stream.synchronize()
        B.tqfx4_check(wsh)
        assert torch.equal(oh.view(torch.int32), ref.view(torch.int32)), t


def test_moe_top_k_equals_n_experts():
    layer = MoeLayer.synthetic(3, 4, 256, 256, 4, 0.0, DEV)
    run_and_check(layer, 3, inputs.hidden_states(3, 2, 256))


def test_moe_argument_errors(full_layer):
    ws = full_layer.workspace(1)
    x = torch.zeros(4096, device=DEV)
    with pytest.raises(B.TqfxError) as e:
        full_layer.ffn(x, ws[:1024])
    assert e.value.status == 4
    bad = B.c_router(full_layer.router_w, None, 0)
    with pytest.raises(B.TqfxError) as e:
        B.tqfx4_moe_ffn(full_layer.ex, bad, x, x, torch.zeros(8, dtype=torch.int32, device=DEV),
                        torch.zeros(8, device=DEV), ws)
    assert e.value.status == 2
    with pytest.raises(B.TqfxError) as e:
        full_layer.ffn(x[1:], ws)
    assert e.value.status == 3


def test_expert_ffn_equals_the_one_expert_layer():
    # tqfx4_expert_ffn (no router) against tqfx4_moe_ffn on the same expert as
    # a one-expert layer, and against the oracle: output and intermediates
    layer = MoeLayer.synthetic(2, 1, 4096, 2048, 1, 0.0, DEV)
    X = inputs.hidden_states(2, 3, 4096)
    ws_moe = layer.workspace(1)
    ws_exp = layer.expert_workspace()
    ex = oracle_experts(2, [0], 4096, 2048)
    for t in range(3):
        x = X[t].to(DEV)
        out_moe = layer.ffn(x, ws_moe)[0].clone()
        out_exp = layer.expert_ffn(0, x, ws_exp)
        B.tqfx4_check(ws_moe)
        B.tqfx4_check(ws_exp)
        assert torch.equal(out_exp.view(torch.int32), out_moe.view(torch.int32))
        for name, dt, shape in (("qx", torch.int8, (4096,)), ("g", torch.float32, (2048,)),
                                ("u", torch.float32, (2048,)), ("h", torch.float32, (2048,)),
                                ("qh", torch.int8, (2048,)), ("o", torch.float32, (4096,))):
            a_ = layer.view(ws_moe, name, dt, shape)
            b_ = layer.view(ws_exp, name, dt, shape)
            assert torch.equal(a_.view(torch.uint8), b_.view(torch.uint8)), name
        ref, _ = oracle.expert_ffn(*ex[0], 4096, 2048, X[t].numpy())
        assert np.array_equal(out_exp.cpu().numpy().view(np.uint32), ref.view(np.uint32))


@pytest.mark.parametrize("H,I", [(1024, 512), (2048, 4096), (768, 1280)])
def test_expert_ffn_of_one_expert_of_a_layer(H, I):
    # expert 5 of an 8-expert layer, ragged block counts, 20 calls in a row
    # on one workspace (gate/up's unit counter is reset by every call)
    layer = MoeLayer.synthetic(H + I, 8, H, I, 2, 0.0, DEV)
    ws = layer.expert_workspace()
    ex = oracle_experts(H + I, [5], H, I)
    X = inputs.hidden_states(H, 2, H)
    refs = [oracle.expert_ffn(*ex[5], H, I, X[t].numpy())[0] for t in range(2)]
    for c in range(20):
        out = layer.expert_ffn(5, X[c % 2].to(DEV), ws)
        B.tqfx4_check(ws)
        assert np.array_equal(out.cpu().numpy().view(np.uint32), refs[c % 2].view(np.uint32))


@pytest.mark.parametrize("H,I,launches", [(4096, 2048, 1), (768, 1280, 2)])
def test_expert_ffn_traced_and_its_launch_count(H, I, launches):
    # the traced call (three events on the stream) gives the untraced call's
    # bits on both paths, and the launch-count query names the path
    assert B.tqfx4_expert_ffn_launches(H, I) == launches
    layer = MoeLayer.synthetic(H + 7, 1, H, I, 1, 0.0, DEV)
    ws = layer.expert_workspace()
    x = inputs.hidden_states(H + 7, 1, H)[0].to(DEV)
    ref = layer.expert_ffn(0, x, ws).clone()
    ev = [torch.cuda.Event(enable_timing=True) for _ in range(3)]
    for e in ev:  # torch creates an event's handle at its first record
        e.record()
    torch.cuda.synchronize()
    out = layer.expert_ffn(0, x, ws, events=ev)
    torch.cuda.synchronize()
    B.tqfx4_check(ws)
    assert torch.equal(out.view(torch.int32), ref.view(torch.int32))
    assert ev[0].elapsed_time(ev[1]) > 0.0 and ev[1].elapsed_time(ev[2]) >= 0.0


def test_expert_ffn_reports_nonfinite_input():
    layer = MoeLayer.synthetic(4, 1, 1024, 512, 1, 0.0, DEV)
    ws = layer.expert_workspace()
    x = inputs.hidden_states(4, 1, 1024)[0]
    x[5] = float("nan")
    layer.expert_ffn(0, x.to(DEV), ws)
    with pytest.raises(B.TqfxError) as e:
        B.tqfx4_check(ws)
    assert e.value.status == 7
