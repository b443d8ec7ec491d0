"""An expert tier for one-token MoE decode: every expert's blocks live in
pinned host memory, and a slab of device slots holds the experts that recent
tokens used (least recently used replaced first). A token is routed on the
GPU (tqfx4_moe_route), the selection is read on the host, each missing
expert is copied into a slot as one contiguous range (its gate, up and down
blocks stored back to back, in host memory and in the slot: the paper's
"one contiguous read per miss" of its streamed store, Sec. 2.2), and
tqfx4_moe_experts runs the expert projections on the slots. The bytes and
kernels are the resident path's, so the outputs equal tqfx4_moe_ffn's bit
for bit wherever an expert was cached.

Plumbing only: copies are cudaMemcpyAsync (torch copy_ from pinned memory)
on the caller's stream, all compute is in the library's kernels.
"""
from collections import OrderedDict

import torch

from . import binding as B


class ExpertTier:
    def __init__(self, layer, slots: int, device=None):
        """layer: a MoeLayer (its blocks are copied to pinned host memory,
        expert by expert; the layer's own device copy is not used by the
        tier). slots: device expert slots, at least top_k."""
        if slots < layer.top_k:
            raise ValueError("the slab needs at least top_k slots")
        self.layer = layer
        dev = device or layer.gate.device
        E, mg, md = layer.n_experts, layer.mb_gu, layer.mb_d
        self.expert_bytes = 2 * mg + md
        # one contiguous range per expert: gate | up | down
        per = torch.cat([layer.gate.view(E, mg), layer.up.view(E, mg), layer.down.view(E, md)], dim=1)
        self.host = per.cpu().pin_memory()
        del per
        self.slab = torch.empty((slots, self.expert_bytes), dtype=torch.uint8, device=dev)
        self.offsets = (0, mg, 2 * mg)  # gate, up, down within an expert's range
        self.slot_of = OrderedDict()  # expert -> slot, least recently used first
        self.free = list(range(slots))
        K = layer.top_k
        self.ptr_h = torch.empty(3 * K, dtype=torch.int64).pin_memory()
        self.ptr_np = self.ptr_h.numpy()
        self.ptr_d = torch.empty(3 * K, dtype=torch.int64, device=dev)
        self.sel_h = torch.empty(K, dtype=torch.int32).pin_memory()
        self.sel_np = self.sel_h.numpy()
        self.slab_base = self.slab.data_ptr()
        self.misses = 0
        self.lookups = 0

    def _slot(self, e: int, keep):
        self.lookups += 1
        s = self.slot_of.get(e)
        if s is not None:
            self.slot_of.move_to_end(e)
            return s
        self.misses += 1
        if self.free:
            s = self.free.pop()
        else:  # the least recently used expert that this token does not need
            victim = next(v for v in self.slot_of if v not in keep)
            s = self.slot_of.pop(victim)
        self.slab[s].copy_(self.host[e], non_blocking=True)
        self.slot_of[e] = s
        return s

    def ffn(self, x, ws, out, sel_idx, sel_w, stream=None):
        """Runs on `stream` (default: the current stream)."""
        st = stream or torch.cuda.current_stream(x.device)
        with torch.cuda.stream(st):
            return self._ffn(x, ws, out, sel_idx, sel_w, st)

    def _ffn(self, x, ws, out, sel_idx, sel_w, st):
        L = self.layer
        B.tqfx4_moe_route(L.ex, L.rt, x, sel_idx, sel_w, ws, st)
        self.sel_h.copy_(sel_idx, non_blocking=True)
        st.synchronize()  # the host needs the selection to place the experts
        sel = self.sel_np.tolist()
        keep = set(sel)
        K = L.top_k
        for j, e in enumerate(sel):
            base = self.slab_base + self._slot(e, keep) * self.expert_bytes
            for p, off in enumerate(self.offsets):
                self.ptr_np[p * K + j] = base + off
        self.ptr_d.copy_(self.ptr_h, non_blocking=True)
        B.tqfx4_moe_experts(L.ex, L.rt, self.ptr_d, out, ws, st)
        return out, sel_idx, sel_w
