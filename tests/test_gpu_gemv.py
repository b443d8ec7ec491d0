"""GPU parity of tqfx4_pack, tqfx4_quantize_act and tqfx4_gemv against the
CPU oracle, through the C ABI: blocks, int8 codes and int32 block sums must
be bit-exact; fp32 GEMV outputs follow the same fixed float schedule as the
oracle and are required bit-exact as well (and within 1e-4 relative)."""
import numpy as np
import pytest
import torch

import oracle
from paper_2608_08910_gb300 import binding as B
from paper_2608_08910_gb300 import inputs, ops
from tests.parity import FP32_TOL, rel_err

pytestmark = pytest.mark.gpu

DEV = "cuda"

# (n, k): the 1024x1024 single-GEMV workload, the expert projections, and
# shapes with ragged tails, odd block counts (8-byte aligned stripes), a
# single block, and K > 32 blocks (one row group per unit)
SHAPES = [(4, 256), (1024, 1024), (2048, 4096), (4096, 2048), (132, 768), (260, 1280), (8, 16384),
          (1204, 512), (36, 256 * 33), (12, 256 * 7)]


@pytest.fixture(scope="module")
def ws():
    return ops.workspace(B.TQFX4_STATUS_BYTES)


def _w(n, k, seed):
    return inputs.log_uniform_scale_matrix(seed, n, k)


@pytest.mark.parametrize("n,k", SHAPES)
def test_pack_rtn_bit_exact(n, k, ws):
    w = _w(n, k, n + k)
    ref = oracle.pack_rtn(w.numpy())
    got = ops.pack_rtn(w.to(DEV), ws).cpu().numpy()
    B.tqfx4_check(ws)
    assert np.array_equal(got, ref)


def test_pack_rtn_student_t_expert_bit_exact(ws):
    w = inputs.expert_matrix(0, 3, inputs.PROJ_GATE, 4096, 2048)
    assert np.array_equal(ops.pack_rtn(w.to(DEV), ws).cpu().numpy(), oracle.pack_rtn(w.numpy()))


@pytest.mark.parametrize("n,k", [(4, 256), (64, 1024), (132, 768), (2048, 4096)])
def test_pack_trits_bit_exact(n, k, ws):
    t1, t2, s = inputs.trit_planes(n + k, n, k)
    ref = oracle.pack_trits(t1.numpy(), t2.numpy(), s.view(torch.int16).numpy().view(np.uint16))
    got = ops.pack_trits(t1.to(DEV), t2.to(DEV), s.to(DEV), ws).cpu().numpy()
    B.tqfx4_check(ws)
    assert np.array_equal(got, ref)


def test_pack_reports_bad_trit_and_nonfinite(ws):
    t1, t2, s = inputs.trit_planes(5, 8, 512)
    t2[3, 300] = 2
    ops.pack_trits(t1.to(DEV), t2.to(DEV), s.to(DEV), ws)
    with pytest.raises(B.TqfxError) as e:
        B.tqfx4_check(ws)
    assert e.value.status == 7
    w = torch.zeros(8, 256)
    w[1, 1] = float("nan")
    ops.pack_rtn(w.to(DEV), ws)
    with pytest.raises(B.TqfxError):
        B.tqfx4_check(ws)
    B.tqfx4_check(ws)  # cleared


@pytest.mark.parametrize("m,k", [(1, 256), (1, 4096), (3, 2048), (64, 4096), (7, 256 * 33)])
def test_quantize_act_bit_exact(m, k, ws):
    x = inputs.hidden_states(m + k, m, k) * 3.0
    x[0, :256] = 0.0  # an all-zero block
    q, da, bs = ops.quantize_act(x.to(DEV), ws)
    B.tqfx4_check(ws)
    rq, rda, rbs = oracle.quantize_act(x.numpy())
    assert np.array_equal(q.cpu().numpy(), rq)
    assert np.array_equal(da.cpu().numpy().view(np.uint32), rda.view(np.uint32))
    assert np.array_equal(bs.cpu().numpy(), rbs)


def test_quantize_act_reports_nonfinite(ws):
    x = torch.ones(2, 512)
    x[1, 400] = float("inf")
    ops.quantize_act(x.to(DEV), ws)
    with pytest.raises(B.TqfxError):
        B.tqfx4_check(ws)


@pytest.mark.parametrize("n,k", SHAPES)
def test_gemv_block_sums_and_outputs(n, k, ws):
    w = _w(n, k, 3 * n + k)
    x = inputs.hidden_states(n * 7 + k, 1, k)[0]
    blocks_ref = oracle.pack_rtn(w.numpy())
    rq, rda, rbs = oracle.quantize_act(x.numpy())
    ry, rS = oracle.gemv(blocks_ref, n, k, rq, rda)
    blocks = ops.pack_rtn(w.to(DEV), ws)
    q, da, bs = ops.quantize_act(x.to(DEV), ws)
    y, S = ops.gemv(blocks, n, k, q, da, bs, ws, block_sums=True)
    B.tqfx4_check(ws)
    assert np.array_equal(S.cpu().numpy(), rS)
    yg = y.cpu().numpy()
    assert rel_err(yg, ry) <= FP32_TOL
    assert np.array_equal(yg.view(np.uint32), ry.view(np.uint32))  # same float schedule


def test_gemv_without_block_sums_matches(ws):
    n, k = 2048, 4096
    w = _w(n, k, 11)
    x = inputs.hidden_states(12, 1, k)[0]
    blocks = ops.pack_rtn(w.to(DEV), ws)
    q, da, bs = ops.quantize_act(x.to(DEV), ws)
    y1, _ = ops.gemv(blocks, n, k, q, da, bs, ws, block_sums=True)
    y2 = ops.gemv(blocks, n, k, q, da, bs, ws)
    assert torch.equal(y1, y2)


def test_gemv_is_independent_of_where_the_bytes_sit(ws):
    # Sec. 2.2: resident and streamed copies are the same bytes, so outputs
    # must not depend on the address the blocks are read from.
    n, k = 1024, 1024
    w = _w(n, k, 21)
    x = inputs.hidden_states(22, 1, k)[0]
    blocks = ops.pack_rtn(w.to(DEV), ws)
    q, da, bs = ops.quantize_act(x.to(DEV), ws)
    y0 = ops.gemv(blocks, n, k, q, da, bs, ws)
    big = torch.zeros(blocks.numel() + 4096, dtype=torch.uint8, device=DEV)
    for off in (16, 48, 1040, 4096):
        view = big[off:off + blocks.numel()]
        view.copy_(blocks)
        assert torch.equal(ops.gemv(view, n, k, q, da, bs, ws), y0)
    assert torch.equal(ops.gemv(blocks, n, k, q, da, bs, ws), y0)  # repeatable


def test_gemv_degenerate_sizes(ws):
    q = torch.zeros(0, dtype=torch.int8, device=DEV)
    f = torch.zeros(0, dtype=torch.float32, device=DEV)
    i = torch.zeros(0, dtype=torch.int32, device=DEV)
    y = torch.full((8,), 5.0, device=DEV)
    B.tqfx4_gemv(torch.zeros(16, dtype=torch.uint8, device=DEV), 8, 0, q, f, i, y, None, ws)
    assert torch.all(y == 0)
    B.tqfx4_gemv(None, 0, 256, q, f, i, y, None, ws)  # n == 0: nothing to do
    B.tqfx4_check(ws)


def test_host_side_argument_errors(ws):
    blocks = torch.zeros(1040, dtype=torch.uint8, device=DEV)
    q = torch.zeros(256, dtype=torch.int8, device=DEV)
    f = torch.zeros(1, device=DEV)
    i = torch.zeros(1, dtype=torch.int32, device=DEV)
    y = torch.zeros(8, device=DEV)
    cases = [
        (lambda: B.tqfx4_gemv(blocks, 6, 256, q, f, i, y, None, ws), 2),
        (lambda: B.tqfx4_gemv(blocks, 8, 100, q, f, i, y, None, ws), 2),
        (lambda: B.tqfx4_gemv(blocks[8:], 8, 256, q, f, i, y, None, ws), 3),
        (lambda: B.tqfx4_gemv(blocks, 8, 256, q, f, i, y, None, ws[:16]), 4),
        (lambda: B.tqfx4_gemv(blocks, 8, 256, q, f, i, None, None, ws), 1),
        (lambda: B.tqfx4_pack(5, blocks, None, None, 8, 256, blocks, ws), 1),
    ]
    for fn, status in cases:
        with pytest.raises(B.TqfxError) as e:
            fn()
        assert e.value.status == status


def test_gemv_large_sampled(ws):
    # 131072 x 4096 (272 MB of blocks, larger than L2): the chunked pass with
    # many more row groups than warps, so each warp carries its ring across
    # row groups. The oracle packs and multiplies sampled row groups (the
    # first and last four and 100 random ones) from the same fp32 rows; the
    # GPU's blocks of those row groups and their outputs must be bit-exact.
    n, k = 131072, 4096
    w = inputs.gemv_matrix(3, n, k, DEV)
    blocks = ops.pack_rtn(w, ws)
    x = inputs.hidden_states(4, 1, k)[0]
    q, da, bs = ops.quantize_act(x.to(DEV), ws)
    y = ops.gemv(blocks, n, k, q, da, bs, ws)
    B.tqfx4_check(ws)
    groups = np.unique(np.concatenate([np.arange(4), np.arange(n // 4 - 4, n // 4),
                                       np.random.default_rng(1).integers(0, n // 4, 100)]))
    rows = (groups[:, None] * 4 + np.arange(4)[None, :]).reshape(-1)
    w_rows = w[torch.from_numpy(rows).to(DEV)].cpu().numpy()
    del w
    ref_blocks = oracle.pack_rtn(w_rows)
    gb = B.tqfx4_matrix_bytes(4, k)
    got_blocks = blocks.view(n // 4, gb)[torch.from_numpy(groups).to(DEV)].cpu().numpy().reshape(-1)
    assert np.array_equal(got_blocks, ref_blocks)
    rq, rda, rbs = oracle.quantize_act(x.numpy())
    assert np.array_equal(q.cpu().numpy(), rq) and np.array_equal(bs.cpu().numpy(), rbs)
    ry, _ = oracle.gemv(ref_blocks, len(rows), k, rq, rda)
    assert np.array_equal(y.cpu().numpy()[rows].view(np.uint32), ry.view(np.uint32))


def test_gemv_1024_benchmark_inputs(ws):
    # the single-GEMV workload's own inputs: N(0, 0.02) weights, seed 0,
    # round-to-nearest codes; an N(0, 1) vector quantized per block
    n = k = 1024
    w = inputs.gemv_matrix(0, n, k)
    x = inputs.hidden_states(0, 1, k)[0]
    rb = oracle.pack_rtn(w.numpy())
    rq, rda, _ = oracle.quantize_act(x.numpy())
    ry, rS = oracle.gemv(rb, n, k, rq, rda)
    blocks = ops.pack_rtn(w.to(DEV), ws)
    q, da, bs = ops.quantize_act(x.to(DEV), ws)
    y, S = ops.gemv(blocks, n, k, q, da, bs, ws, block_sums=True)
    B.tqfx4_check(ws)
    assert np.array_equal(blocks.cpu().numpy(), rb)
    assert np.array_equal(S.cpu().numpy(), rS)
    assert np.array_equal(y.cpu().numpy().view(np.uint32), ry.view(np.uint32))
    assert rel_err(y.cpu().numpy(), ry) <= FP32_TOL


# the one-launch GEMV (quantization inside): shapes of the chunked pass with
# ragged row counts, 2 to 64 blocks a row, more row groups than warps
SHAPES_X = [(4, 512), (1024, 1024), (260, 4096), (2048, 4096), (4096, 2048), (12, 8192), (1204, 512),
            (8, 16384), (16388, 1024)]


@pytest.mark.parametrize("n,k", SHAPES_X)
def test_gemv_x_equals_quantize_then_gemv(n, k, ws):
    w = _w(n, k, 3 * n + k)
    x = inputs.hidden_states(n + k, 1, k)[0].to(DEV)
    blocks = ops.pack_rtn(w.to(DEV), ws)
    q, da, bs = ops.quantize_act(x, ws)
    y = ops.gemv(blocks, n, k, q, da, bs, ws)
    y2, q2, da2, bs2 = ops.gemv_x(blocks, n, k, x, ws, quantized=True)
    y3 = ops.gemv_x(blocks, n, k, x, ws)
    B.tqfx4_check(ws)
    assert torch.equal(q2, q) and torch.equal(bs2, bs)
    assert torch.equal(da2.view(torch.int32), da.view(torch.int32))
    assert torch.equal(y2.view(torch.int32), y.view(torch.int32))
    assert torch.equal(y3.view(torch.int32), y.view(torch.int32))


def test_gemv_x_1024_benchmark_inputs(ws):
    # the single-GEMV workload in one launch, against the oracle
    n = k = 1024
    w = inputs.gemv_matrix(0, n, k)
    x = inputs.hidden_states(0, 1, k)[0]
    rb = oracle.pack_rtn(w.numpy())
    rq, rda, rbs = oracle.quantize_act(x.numpy())
    ry, _ = oracle.gemv(rb, n, k, rq, rda)
    blocks = ops.pack_rtn(w.to(DEV), ws)
    y, q, da, bs = ops.gemv_x(blocks, n, k, x.to(DEV), ws, quantized=True)
    B.tqfx4_check(ws)
    assert np.array_equal(q.cpu().numpy(), rq.reshape(-1))
    assert np.array_equal(da.cpu().numpy().view(np.uint32), rda.reshape(-1).view(np.uint32))
    assert np.array_equal(bs.cpu().numpy(), rbs.reshape(-1))
    assert np.array_equal(y.cpu().numpy().view(np.uint32), ry.view(np.uint32))
    assert rel_err(y.cpu().numpy(), ry) <= FP32_TOL


def _host(v, kind):
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
@pytest.mark.parametrize("n,k", [(1024, 1024), (2048, 4096), (36, 512)])
def test_gemv_x_host_equals_the_device_call(n, k, kind, ws):
    # x and y in host memory (page-locked ones used in place by the kernel,
    # the others through staging copies): y bit-identical to gemv_x's
    blocks = ops.pack_rtn(_w(n, k, 5 * n + k).to(DEV), ws)
    wsh = ops.gemv_x_host_workspace(n, k)
    stream = torch.cuda.current_stream()
    for t in range(3):
        x = inputs.hidden_states(n + k + t, 1, k)[0]
        ref = ops.gemv_x(blocks, n, k, x.to(DEV), ws).cpu()
        xh, yh = _host(x, kind), _host(torch.zeros(n), kind)
        ops.gemv_x_host(blocks, n, k, xh, yh, wsh, stream)
        stream.synchronize()
        B.tqfx4_check(wsh)
        assert torch.equal(yh.view(torch.int32), ref.view(torch.int32)), t


def test_gemv_x_reports_nonfinite_activation(ws):
    n, k = 64, 1024
    blocks = ops.pack_rtn(_w(n, k, 1).to(DEV), ws)
    x = inputs.hidden_states(1, 1, k)[0]
    x[700] = float("inf")
    ops.gemv_x(blocks, n, k, x.to(DEV), ws)
    with pytest.raises(B.TqfxError) as e:
        B.tqfx4_check(ws)
    assert e.value.status == 7
