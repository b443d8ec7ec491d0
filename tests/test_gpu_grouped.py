"""GPU parity of tqfx4_moe_grouped (T tokens grouped by expert: batched
decode and prefill) against the CPU oracle, through the C ABI, on every
contraction: the decode path (legacy integer MMA), the prefill path (tcgen05
tensor cores on exact e4m3 encodings of the codes and of the two activation
planes; chunks of at most 4 pairs stream through the integer small-group
pass) and the automatic choice (the prefill path).

Per call: the routing of every token (bit-exact up to accepted near-ties),
the grouping (counts, offsets and the stable expert-then-token order,
bit-exact against the oracle's counting sort), and for sampled tokens the
per-pair g, u, quantized h and expert outputs (bit-exact) and the combined
output (within 1e-4 relative; equal to tqfx4_moe_ffn on the same token).
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


def run_grouped(layer, X, path=0):
    T = X.shape[0]
    ws = layer.workspace(T, path)
    OUT, sel, selw = layer.grouped(X.to(DEV), ws, path)
    B.tqfx4_check(ws)
    return ws, OUT.cpu().numpy(), sel.cpu().numpy(), selw.cpu().numpy()


def check_grouped(layer, seed, X, sample, path=0, check_stages=True, stage_tokens=None):
    """Checks the call's routing and grouping for every token, the combined
    output of the `sample` tokens against the oracle, and, for the
    `stage_tokens` (default: the sample, if check_stages), every pair's g,
    u, quantized h and expert output bit for bit. Returns (OUT, sel, selw,
    near-tie count, the stage-checked (token, expert) pairs)."""
    H, I, E, k = layer.hidden, layer.inter, layer.n_experts, layer.top_k
    T = X.shape[0]
    P = T * k
    ws, OUT, sel, selw = run_grouped(layer, X, path)
    Wr = layer.router_w.cpu().numpy()
    bias = None if layer.router_b is None else layer.router_b.cpu().numpy()
    Xn = X.numpy()
    ties = 0
    for t in range(T):
        logits, r_idx, r_w = oracle.router(Wr, bias, Xn[t], k)
        n = check_selection(sel[t], logits, selection_tolerance(Wr, Xn[t], bias), k)
        ties += n
        if n == 0:
            assert np.allclose(selw[t], r_w, rtol=1.2e-7, atol=0)
    # grouping: the oracle's stable counting sort of the kernel's own selection
    counts, offsets, pt, ps = oracle.group_by_expert(sel, E)
    g = lambda name, dt, shape: layer.view(ws, name, dt, shape, tokens=T, grouped=1, path=path).cpu().numpy()
    assert np.array_equal(g("counts", torch.int32, (E,)), counts)
    assert np.array_equal(g("offsets", torch.int32, (E + 1,)), offsets)
    assert np.array_equal(g("pair_token", torch.int32, (P,)), pt)
    assert np.array_equal(g("pair_slot", torch.int32, (P,)), ps)
    pair_of = g("pair_of", torch.int32, (T, k))
    assert np.array_equal(pt[pair_of], np.repeat(np.arange(T), k).reshape(T, k))
    if stage_tokens is None:
        stage_tokens = sample if check_stages else []
    elif callable(stage_tokens):
        stage_tokens = stage_tokens(sel)
    if len(stage_tokens):
        gv, uv = g("g", torch.float32, (P, I)), g("u", torch.float32, (P, I))
        qh, ov = g("qh", torch.int8, (P, I)), g("o", torch.float32, (P, H))
    checked = []
    hits = np.bincount(sel.ravel(), minlength=E)
    for t in sorted(set(sample) | set(stage_tokens)):
        ex = oracle_experts(seed, sel[t], H, I)
        if t in stage_tokens:  # stage by stage first: a failure names the stage and the pair
            for j in range(k):
                pos = pair_of[t, j]
                e = int(sel[t, j])
                ro, dbg = oracle.expert_ffn(*ex[e], H, I, Xn[t])
                where = "token %d slot %d expert %d (%d pairs)" % (t, j, e, hits[e])
                for name, got, want in (("g", gv[pos], dbg["g"]), ("u", uv[pos], dbg["u"]),
                                        ("qh", qh[pos], dbg["qh"]), ("o", ov[pos], ro)):
                    gb = got.view(np.uint32) if got.dtype == np.float32 else got
                    wb = want.view(np.uint32) if want.dtype == np.float32 else want
                    bad = np.flatnonzero(gb != wb)
                    assert bad.size == 0, "%s: %s differs at %d of %d entries (first %s)" % (
                        where, name, bad.size, got.size, bad[:8])
                checked.append((t, e))
        if t in sample:
            ref, ridx, _ = oracle.moe_tokens(ex, E, H, I, Wr, bias, k, Xn[t])
            if np.array_equal(ridx[0], sel[t]):
                e_ = rel_err(OUT[t], ref[0])
                assert e_ <= FP32_TOL, (t, e_)
    return OUT, sel, selw, ties, checked


@pytest.mark.parametrize("E,H,I,k,T,zipf", [
    (16, 512, 1024, 4, 20, 0.0),     # ragged counts, one chunk per expert
    (8, 512, 512, 4, 200, 0.0),      # ~100 pairs per expert: two chunks, ragged tail
    (32, 1024, 512, 6, 33, 1.1),     # skewed routing
    (4, 512, 512, 4, 3, 0.0),        # top_k = n_experts
    (64, 2048, 1536, 8, 1, 0.0),     # a single token; inter not a multiple of 1024
    (512, 512, 512, 8, 600, 1.1),    # 10-bit expert indices; 4800 pairs: the wide (token, slot) scatter
])
@pytest.mark.parametrize("path", [B.TQFX4_PATH_DECODE, B.TQFX4_PATH_PREFILL])
def test_grouped_small(E, H, I, k, T, zipf, path):
    seed = 100 + E + T
    layer = MoeLayer.synthetic(seed, E, H, I, k, zipf, DEV)
    X = inputs.hidden_states(seed, T, H)
    check_grouped(layer, seed, X, sample=range(min(T, 6)), path=path)


@pytest.mark.parametrize("path", [B.TQFX4_PATH_DECODE, B.TQFX4_PATH_PREFILL])
def test_grouped_equals_per_token_moe_ffn(path):
    layer = MoeLayer.synthetic(5, 32, 1024, 1024, 8, 0.0, DEV)
    X = inputs.hidden_states(5, 24, 1024)
    ws, OUT, sel, selw = run_grouped(layer, X, path)
    wsd = layer.workspace(1)
    for t in range(24):
        out, s, w = layer.ffn(X[t].to(DEV), wsd)
        assert np.array_equal(s.cpu().numpy(), sel[t])
        assert np.array_equal(w.cpu().numpy(), selw[t])
        assert np.array_equal(out.cpu().numpy().view(np.uint32), OUT[t].view(np.uint32))


def test_tensor_core_path_equals_integer_mma_path():
    # every pair's g, u, quantized h and expert output, and the combined
    # output, bit-identical between the two contractions: ~150 pairs per
    # expert (three chunks, ragged), 8 row tiles of 128 rows, ragged tiles
    E, H, I, k, T = 16, 1536, 1024, 4, 600
    layer = MoeLayer.synthetic(8, E, H, I, k, 0.5, DEV)
    X = inputs.hidden_states(8, T, H)
    P = T * k
    res = []
    for path in (B.TQFX4_PATH_DECODE, B.TQFX4_PATH_PREFILL):
        ws, OUT, sel, selw = run_grouped(layer, X, path)
        g = lambda name, dt, shape: layer.view(ws, name, dt, shape, tokens=T, grouped=1, path=path).cpu().numpy()
        res.append([OUT, sel, g("g", torch.float32, (P, I)), g("u", torch.float32, (P, I)),
                    g("qh", torch.int8, (P, I)), g("o", torch.float32, (P, H))])
    for a, b in zip(*res):
        assert np.array_equal(a.view(np.uint8), b.view(np.uint8))


@pytest.mark.parametrize("kind", ["pinned", "pageable"])
@pytest.mark.parametrize("path", [B.TQFX4_PATH_DECODE, B.TQFX4_PATH_PREFILL])
def test_grouped_host_equals_the_device_call(kind, path):
    # X, OUT and the selection in host memory (page-locked ones used in place:
    # a copy kernel reads X, the combine and the top-k write into host memory;
    # pageable ones through staging copies): the device call's bits
    layer = MoeLayer.synthetic(12, 32, 1024, 512, 6, 1.1, DEV)
    T = 40
    X = inputs.hidden_states(12, T, 1024)
    ws = layer.workspace(T, path)
    OUT, sel, selw = layer.grouped(X.to(DEV), ws, path)
    wsh = layer.grouped_host_workspace(T, path)
    host = (lambda t: t.pin_memory()) if kind == "pinned" else (lambda t: t)
    Xh = host(X.clone())
    OUTh = host(torch.zeros(T, 1024))
    selh, selwh = host(torch.zeros(T, 6, dtype=torch.int32)), host(torch.zeros(T, 6))
    stream = torch.cuda.current_stream()
    layer.grouped_host(Xh, wsh, OUTh, selh, selwh, path, stream=stream)
    stream.synchronize()
    B.tqfx4_check(wsh)
    assert torch.equal(OUTh.view(torch.int32), OUT.cpu().view(torch.int32))
    assert torch.equal(selh, sel.cpu())
    assert torch.equal(selwh.view(torch.int32), selw.cpu().view(torch.int32))


def test_grouped_empty_batch():
    layer = MoeLayer.synthetic(6, 8, 512, 512, 2, 0.0, DEV)
    ws = layer.workspace(1)
    X = torch.zeros((0, 512), device=DEV)
    OUT = torch.zeros((0, 512), device=DEV)
    B.tqfx4_moe_grouped(layer.ex, layer.rt, X, 0, OUT, torch.zeros(0, dtype=torch.int32, device=DEV),
                        torch.zeros(0, device=DEV), 0, ws)
    B.tqfx4_check(ws)


def test_grouped_rejects_odd_block_counts():
    layer = MoeLayer.synthetic(6, 8, 768, 512, 2, 0.0, DEV)  # hidden = 3 blocks
    X = inputs.hidden_states(6, 2, 768).to(DEV)
    ws = torch.zeros(1 << 20, dtype=torch.uint8, device=DEV)
    with pytest.raises(B.TqfxError) as e:
        layer.grouped(X, ws)
    assert e.value.status == 2


@pytest.fixture(scope="module")
def zipf_layer():
    return MoeLayer.synthetic(0, 256, 4096, 2048, 8, 1.1, DEV)


def test_grouped_decode_64_tokens_zipf_full_size(zipf_layer):
    # batched decode: 64 tokens, 256 experts, top-8, Zipf(1.1) router bias
    X = inputs.hidden_states(0, 64, 4096)
    OUT, sel, selw, ties, _ = check_grouped(zipf_layer, 0, X, sample=[0, 17, 63], path=B.TQFX4_PATH_DECODE)
    hits = np.bincount(sel.ravel(), minlength=256)
    assert hits.max() > 8 and (hits > 0).sum() < 256  # the skew is visible


def test_grouped_decode_64_tokens_zipf_full_size_auto(zipf_layer):
    # the batched-decode workload on the path the library chooses (AUTO):
    # experts with at most 4 pairs go through the streaming small-group pass
    # at K = 4096 (gate/up) and K = 2048 (down), the others through the
    # tensor-core contraction. Every token's routing and the grouping are
    # checked; 8 tokens' outputs against the oracle; every pair of 4 tokens
    # stage by stage (g, u, quantized h, expert output), bit for bit.
    X = inputs.hidden_states(0, 64, 4096)
    sample = [0, 5, 17, 26, 31, 40, 52, 63]

    def stage_tokens(sel):
        # token 0 and the three tokens with the most pairs on experts of at
        # most 4 pairs (the small-group pass)
        hits = np.bincount(sel.ravel(), minlength=256)
        n_small = (hits[sel] <= 4).sum(axis=1)
        return sorted({0, *np.argsort(-n_small, kind="stable")[:3].tolist()})

    OUT, sel, selw, ties, checked = check_grouped(zipf_layer, 0, X, sample=sample, path=B.TQFX4_PATH_AUTO,
                                                  stage_tokens=stage_tokens)
    hits = np.bincount(sel.ravel(), minlength=256)
    small = [e for _, e in checked if hits[e] <= 4]
    tensor = [e for _, e in checked if hits[e] > 4]
    assert len(small) >= 4 and len(tensor) >= 4, (len(small), len(tensor))  # both contractions covered

@pytest.fixture(scope="module")
def prefill_layer():
    return MoeLayer.synthetic(0, 256, 4096, 2048, 8, 0.0, DEV)


def test_grouped_prefill_2048_tokens_full_size(prefill_layer):
    # every token's routing and the grouping; 3 tokens' outputs, and every
    # pair of 2 of them stage by stage, on the tensor-core contraction at
    # K = 4096 / 2048 (about 64 pairs a chunk)
    X = inputs.hidden_states(1, 2048, 4096)
    check_grouped(prefill_layer, 0, X, sample=[0, 1023, 2047], path=B.TQFX4_PATH_PREFILL,
                  stage_tokens=[1023, 2047])
