"""Tensor-allocating conveniences over the C ABI (binding.py).

Each helper allocates its outputs with torch on the inputs' device and makes
exactly one library call; none computes anything itself.
"""
import torch

from . import binding as B


def workspace(nbytes: int, device="cuda") -> torch.Tensor:
    """Zeroed device workspace (torch allocations are 256-byte aligned)."""
    n = max(int(nbytes), B.TQFX4_STATUS_BYTES)
    return torch.zeros(((n + 255) // 256) * 256, dtype=torch.uint8, device=device)


def empty_blocks(n: int, k: int, device="cuda", count: int = 1) -> torch.Tensor:
    nbytes = B.tqfx4_matrix_bytes(n, k)
    if nbytes < 0:
        raise ValueError("bad shape %dx%d" % (n, k))
    return torch.empty(count * nbytes, dtype=torch.uint8, device=device)


def pack_rtn(w: torch.Tensor, ws: torch.Tensor, out: torch.Tensor = None) -> torch.Tensor:
    n, k = w.shape
    blocks = empty_blocks(n, k, w.device) if out is None else out
    B.tqfx4_pack(B.TQFX4_SRC_F32_RTN, w, None, None, n, k, blocks, ws)
    return blocks


def pack_tied(w: torch.Tensor, ws: torch.Tensor, out: torch.Tensor = None) -> torch.Tensor:
    n, k = w.shape
    blocks = empty_blocks(n, k, w.device) if out is None else out
    B.tqfx4_pack(B.TQFX4_SRC_F32_TIED, w, None, None, n, k, blocks, ws)
    return blocks


def pack_trits(t1, t2, scales_f16, ws) -> torch.Tensor:
    n, k = t1.shape
    blocks = empty_blocks(n, k, t1.device)
    B.tqfx4_pack(B.TQFX4_SRC_TRITS, t1, t2, scales_f16, n, k, blocks, ws)
    return blocks


def quantize_act(x: torch.Tensor, ws: torch.Tensor):
    x2 = x.reshape(-1, x.shape[-1])
    m, k = x2.shape
    q = torch.empty((m, k), dtype=torch.int8, device=x.device)
    da = torch.empty((m, k // 256), dtype=torch.float32, device=x.device)
    bs = torch.empty((m, k // 256), dtype=torch.int32, device=x.device)
    B.tqfx4_quantize_act(x2, m, k, q, da, bs, ws)
    if x.dim() == 1:
        return q[0], da[0], bs[0]
    return q, da, bs


def gemv(blocks, n: int, k: int, q, da, bsum, ws, block_sums: bool = False):
    y = torch.empty(n, dtype=torch.float32, device=blocks.device)
    S = torch.empty((n, k // 256), dtype=torch.int32, device=blocks.device) if block_sums else None
    B.tqfx4_gemv(blocks, n, k, q, da, bsum, y, S, ws)
    return (y, S) if block_sums else y


def gemv_x_host_workspace(n: int, k: int, device="cuda"):
    """The workspace of gemv_x_host (device memory)."""
    nb = B.tqfx4_gemv_x_host_workspace_bytes(n, k)
    if nb == 0:
        raise ValueError("gemv_x_host: k must be a positive multiple of 512 and n of 4")
    return torch.zeros(nb, dtype=torch.uint8, device=device)


def gemv_x_host(blocks, n: int, k: int, x, y, ws, stream=None):
    """y = W x with x and y in host memory (CPU tensors; page-locked ones are
    used in place); y is complete once `stream` has passed the call."""
    B.tqfx4_gemv_x_host(blocks, n, k, x, y, ws, stream)
    return y


def gemv_x(blocks, n: int, k: int, x, ws, quantized: bool = False):
    """y = W x for an fp32 x, quantized inside the same launch; with
    quantized=True also returns the quantized vector (q, da, bsum)."""
    y = torch.empty(n, dtype=torch.float32, device=blocks.device)
    q = da = bsum = None
    if quantized:
        q = torch.empty(k, dtype=torch.int8, device=blocks.device)
        da = torch.empty(k // 256, dtype=torch.float32, device=blocks.device)
        bsum = torch.empty(k // 256, dtype=torch.int32, device=blocks.device)
    B.tqfx4_gemv_x(blocks, n, k, x, y, q, da, bsum, ws)
    return (y, q, da, bsum) if quantized else y


def gemv_mxfp4(blocks, n: int, k: int, q, da, ws, block_sums: bool = False):
    """y = W x for W in MXFP4 blocks (17 bytes per 32 elements) and x
    quantized by quantize_act."""
    y = torch.empty(n, dtype=torch.float32, device=blocks.device)
    S = torch.empty((n, k // 32), dtype=torch.int32, device=blocks.device) if block_sums else None
    B.tqfx4_gemv_mxfp4(blocks, n, k, q, da, y, S, ws)
    return (y, S) if block_sums else y


def pack_free(t1, t2, a1, a2, ws):
    """Two trit planes int8 [n][k] and their f16 scales [n][k/256] -> blocks
    of the free-scale two-plane format."""
    n, k = t1.shape
    out = torch.empty(B.tqfx4_free_bytes(n, k), dtype=torch.uint8, device=t1.device)
    B.tqfx4_pack_free(t1, t2, a1, a2, n, k, out, ws)
    return out


def gemv_free(blocks, n: int, k: int, q, da, bsum, ws, block_sums: bool = False):
    y = torch.empty(n, dtype=torch.float32, device=blocks.device)
    S1 = S2 = None
    if block_sums:
        S1 = torch.empty((n, k // 256), dtype=torch.int32, device=blocks.device)
        S2 = torch.empty((n, k // 256), dtype=torch.int32, device=blocks.device)
    B.tqfx4_gemv_free(blocks, n, k, q, da, bsum, y, S1, S2, ws)
    return (y, S1, S2) if block_sums else y
