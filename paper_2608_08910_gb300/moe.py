"""A routed-expert MoE layer held in device memory as tq2_0_fx4 blocks (or,
for the expert-lossless arm, as MXFP4 blocks).

Plumbing only: it allocates the stacked expert matrices and the router with
torch, fills them through tqfx4_pack, and calls tqfx4_moe_ffn /
tqfx4_moe_grouped. Each expert projection is one contiguous byte range
(gate and up: inter x hidden; down: hidden x inter), experts stacked in
order, as the C ABI's tqfx4_experts describes.
"""
import torch

from . import binding as B
from . import inputs


class MoeLayer:
    def __init__(self, gate, up, down, router_w, router_b, n_experts, hidden, inter, top_k, fmt="fx4"):
        """fmt: the experts' weight format, "fx4" (tq2_0_fx4 blocks) or
        "mxfp4" (MXFP4 blocks, served by tqfx4_moe_ffn_mxfp4)."""
        self.gate, self.up, self.down = gate, up, down
        self.router_w, self.router_b = router_w, router_b
        self.n_experts, self.hidden, self.inter, self.top_k = n_experts, hidden, inter, top_k
        self.fmt = fmt
        self.ex = B.c_experts(gate, up, down, n_experts, hidden, inter)
        self.rt = B.c_router(router_w, router_b, top_k)
        size = B.tqfx4_mxfp4_bytes if fmt == "mxfp4" else B.tqfx4_matrix_bytes
        self.mb_gu = size(inter, hidden)
        self.mb_d = size(hidden, inter)

    @classmethod
    def synthetic(cls, seed: int, n_experts: int, hidden: int, inter: int, top_k: int, zipf: float = 0.0,
                  device="cuda"):
        """Student-t(5) * 0.02 expert weights packed by round-to-nearest, an
        N(0, 0.02) router, and the -zipf * ln(rank) bias when zipf > 0."""
        mb_gu = B.tqfx4_matrix_bytes(inter, hidden)
        mb_d = B.tqfx4_matrix_bytes(hidden, inter)
        gate = torch.empty(n_experts * mb_gu, dtype=torch.uint8, device=device)
        up = torch.empty(n_experts * mb_gu, dtype=torch.uint8, device=device)
        down = torch.empty(n_experts * mb_d, dtype=torch.uint8, device=device)
        ws = torch.zeros(B.TQFX4_STATUS_BYTES, dtype=torch.uint8, device=device)
        for e in range(n_experts):
            for proj, buf, mb in ((inputs.PROJ_GATE, gate, mb_gu), (inputs.PROJ_UP, up, mb_gu),
                                  (inputs.PROJ_DOWN, down, mb_d)):
                w = inputs.expert_matrix(seed, e, proj, hidden, inter, device)
                n, k = w.shape
                B.tqfx4_pack(B.TQFX4_SRC_F32_RTN, w, None, None, n, k, buf[e * mb:(e + 1) * mb], ws)
        B.tqfx4_check(ws)
        rw = inputs.router_weight(seed, n_experts, hidden, device)
        rb = inputs.zipf_bias(n_experts, zipf).to(device) if zipf > 0 else None
        return cls(gate, up, down, rw, rb, n_experts, hidden, inter, top_k)

    @classmethod
    def synthetic_mxfp4(cls, seed: int, n_experts: int, hidden: int, inter: int, top_k: int, zipf: float = 0.0,
                        device="cuda"):
        """MXFP4 experts (random released-style bytes, inputs.mxfp4_matrix,
        one seed per expert projection) and the router of synthetic()."""
        mb_gu = B.tqfx4_mxfp4_bytes(inter, hidden)
        mb_d = B.tqfx4_mxfp4_bytes(hidden, inter)
        bufs = []
        for proj, (n, k) in ((inputs.PROJ_GATE, (inter, hidden)), (inputs.PROJ_UP, (inter, hidden)),
                             (inputs.PROJ_DOWN, (hidden, inter))):
            bufs.append(torch.cat([inputs.mxfp4_matrix(inputs.expert_seed(seed, e, proj), n, k, device)
                                   for e in range(n_experts)]))
        rw = inputs.router_weight(seed, n_experts, hidden, device)
        rb = inputs.zipf_bias(n_experts, zipf).to(device) if zipf > 0 else None
        return cls(*bufs, rw, rb, n_experts, hidden, inter, top_k, fmt="mxfp4")

    def expert_blocks(self, e: int):
        """The (gate, up, down) byte ranges of expert e."""
        return (self.gate[e * self.mb_gu:(e + 1) * self.mb_gu], self.up[e * self.mb_gu:(e + 1) * self.mb_gu],
                self.down[e * self.mb_d:(e + 1) * self.mb_d])

    def workspace(self, tokens: int = 1, path: int = 0) -> torch.Tensor:
        n = B.tqfx4_moe_workspace_bytes(self.ex, self.rt, tokens, path)
        if n == 0:
            raise ValueError("invalid MoE shapes")
        return torch.zeros(((n + 255) // 256) * 256, dtype=torch.uint8, device=self.gate.device)

    def expert_workspace(self) -> torch.Tensor:
        """A zeroed workspace for expert_ffn."""
        n = B.tqfx4_expert_ffn_workspace_bytes(self.hidden, self.inter)
        if n == 0:
            raise ValueError("invalid expert shapes")
        return torch.zeros(((n + 255) // 256) * 256, dtype=torch.uint8, device=self.gate.device)

    def expert_ffn(self, e: int, x, ws, out=None, stream=None, events=None):
        """Expert e's SwiGLU FFN alone (tqfx4_expert_ffn: no router, weight 1)."""
        if self.fmt != "fx4":
            raise ValueError("expert_ffn serves tq2_0_fx4 experts")
        out = torch.empty(self.hidden, dtype=torch.float32, device=x.device) if out is None else out
        g, u, d = self.expert_blocks(e)
        B.tqfx4_expert_ffn(g, u, d, self.hidden, self.inter, x, out, ws, stream, events)
        return out

    def expert_host_workspace(self) -> torch.Tensor:
        """A zeroed workspace for expert_ffn_host."""
        n = B.tqfx4_expert_ffn_host_workspace_bytes(self.hidden, self.inter)
        if n == 0:
            raise ValueError("invalid expert shapes")
        return torch.zeros(n, dtype=torch.uint8, device=self.gate.device)

    def expert_ffn_host(self, e: int, x, ws, out, stream=None):
        """expert_ffn with x and out in host memory (CPU tensors, page-locked
        ones used in place); out is complete once `stream` has passed it."""
        if self.fmt != "fx4":
            raise ValueError("expert_ffn serves tq2_0_fx4 experts")
        g, u, d = self.expert_blocks(e)
        B.tqfx4_expert_ffn_host(g, u, d, self.hidden, self.inter, x, out, ws, stream)
        return out

    def ffn(self, x, ws, out=None, sel_idx=None, sel_w=None, stream=None, events=None):
        dev = x.device
        out = torch.empty(self.hidden, dtype=torch.float32, device=dev) if out is None else out
        sel_idx = torch.empty(self.top_k, dtype=torch.int32, device=dev) if sel_idx is None else sel_idx
        sel_w = torch.empty(self.top_k, dtype=torch.float32, device=dev) if sel_w is None else sel_w
        if self.fmt == "mxfp4":
            B.tqfx4_moe_ffn_mxfp4(self.ex, self.rt, x, out, sel_idx, sel_w, ws, stream, events)
        else:
            B.tqfx4_moe_ffn(self.ex, self.rt, x, out, sel_idx, sel_w, ws, stream, events)
        return out, sel_idx, sel_w

    def host_workspace(self):
        """The workspace of ffn_host (device memory)."""
        n = B.tqfx4_moe_ffn_host_workspace_bytes(self.ex, self.rt)
        if n == 0:
            raise ValueError("invalid MoE shapes")
        return torch.zeros(n, dtype=torch.uint8, device=self.gate.device)

    def ffn_host(self, x, ws, out, sel_idx=None, sel_w=None, stream=None):
        """One token with x and the outputs in host memory (CPU tensors,
        page-locked for asynchronous copies); ordered on `stream`, complete
        once the stream has passed it."""
        if self.fmt != "fx4":
            raise ValueError("ffn_host serves tq2_0_fx4 experts")
        B.tqfx4_moe_ffn_host(self.ex, self.rt, x, out, sel_idx, sel_w, ws, stream)
        return out, sel_idx, sel_w

    def grouped(self, X, ws, path=0, OUT=None, sel_idx=None, sel_w=None, stream=None, events=None):
        if self.fmt != "fx4":
            raise ValueError("the grouped path serves tq2_0_fx4 experts")
        T = X.shape[0]
        dev = X.device
        OUT = torch.empty((T, self.hidden), dtype=torch.float32, device=dev) if OUT is None else OUT
        sel_idx = torch.empty((T, self.top_k), dtype=torch.int32, device=dev) if sel_idx is None else sel_idx
        sel_w = torch.empty((T, self.top_k), dtype=torch.float32, device=dev) if sel_w is None else sel_w
        B.tqfx4_moe_grouped(self.ex, self.rt, X, T, OUT, sel_idx, sel_w, path, ws, stream, events)
        return OUT, sel_idx, sel_w

    def grouped_host_workspace(self, tokens: int, path: int = 0) -> torch.Tensor:
        """The workspace of grouped_host (device memory)."""
        n = B.tqfx4_moe_grouped_host_workspace_bytes(self.ex, self.rt, tokens, path)
        if n == 0:
            raise ValueError("invalid MoE shapes")
        return torch.zeros(n, dtype=torch.uint8, device=self.gate.device)

    def grouped_host(self, X, ws, OUT, sel_idx=None, sel_w=None, path=0, stream=None):
        """grouped with X and the outputs in host memory (CPU tensors,
        page-locked ones used in place); complete once `stream` has passed it."""
        if self.fmt != "fx4":
            raise ValueError("the grouped path serves tq2_0_fx4 experts")
        B.tqfx4_moe_grouped_host(self.ex, self.rt, X, X.shape[0], OUT, sel_idx, sel_w, path, ws, stream)
        return OUT, sel_idx, sel_w

    def view(self, ws, name, dtype, shape, tokens=1, grouped=0, path=0):
        """A typed view of one intermediate the last call left in `ws`."""
        off = B.tqfx4_moe_workspace_views(self.ex, self.rt, tokens, grouped, path)[name]
        n = 1
        for s in shape:
            n *= s
        nbytes = n * torch.tensor([], dtype=dtype).element_size()
        return ws[off:off + nbytes].view(dtype).view(*shape)
