"""An expert tier for one-token MoE decode: every expert's blocks live in
pinned host memory, and a slab of device slots holds the experts that recent
tokens used (least recently used replaced first). A token is routed on the
GPU (tqfx4_moe_route), the selection is read on the host, each missing
expert's gate, up and down blocks are copied into a slot (one contiguous
range per projection: the "one contiguous read per miss" of the paper's
streamed store, Sec. 2.2), and tqfx4_moe_experts runs the expert
projections on the slots. The bytes and kernels are the resident path's, so
the outputs equal tqfx4_moe_ffn's bit for bit wherever an expert was cached.

Plumbing only: copies are cudaMemcpyAsync (torch copy_ from pinned memory)
on the caller's stream, all compute is in the library's kernels.
"""
from collections import OrderedDict

import torch

from . import binding as B


class ExpertTier:
    def __init__(self, layer, slots: int, device=None):
        """layer: a MoeLayer (its blocks are copied to pinned host memory;
        the layer's own device copy is not used by the tier). slots: device
        expert slots, at least top_k."""
        if slots < layer.top_k:
            raise ValueError("the slab needs at least top_k slots")
        self.layer = layer
        dev = device or layer.gate.device
        E, mg, md = layer.n_experts, layer.mb_gu, layer.mb_d
        self.host = [t.view(E, -1).cpu().pin_memory() for t in (layer.gate, layer.up, layer.down)]
        self.slab = [torch.empty((slots, m), dtype=torch.uint8, device=dev) for m in (mg, mg, md)]
        self.slot_of = OrderedDict()  # expert -> slot, least recently used first
        self.free = list(range(slots))
        K = layer.top_k
        self.ptr_h = torch.empty(3 * K, dtype=torch.int64).pin_memory()
        self.ptr_d = torch.empty(3 * K, dtype=torch.int64, device=dev)
        self.sel_h = torch.empty(K, dtype=torch.int32).pin_memory()
        self.misses = 0
        self.lookups = 0

    def _slot(self, e: int, keep, stream):
        self.lookups += 1
        if e in self.slot_of:
            self.slot_of.move_to_end(e)
            return self.slot_of[e]
        self.misses += 1
        if self.free:
            s = self.free.pop()
        else:  # the least recently used expert that this token does not need
            victim = next(v for v in self.slot_of if v not in keep)
            s = self.slot_of.pop(victim)
        with torch.cuda.stream(stream):
            for slab, host in zip(self.slab, self.host):
                slab[s].copy_(host[e], non_blocking=True)
        self.slot_of[e] = s
        return s

    def ffn(self, x, ws, out, sel_idx, sel_w, stream=None):
        L = self.layer
        st = stream or torch.cuda.current_stream(x.device)
        B.tqfx4_moe_route(L.ex, L.rt, x, sel_idx, sel_w, ws, st)
        with torch.cuda.stream(st):
            self.sel_h.copy_(sel_idx, non_blocking=True)
        st.synchronize()  # the host needs the selection to place the experts
        sel = [int(v) for v in self.sel_h]
        keep = set(sel)
        K = L.top_k
        for j, e in enumerate(sel):
            s = self._slot(e, keep, st)
            for p in range(3):
                self.ptr_h[p * K + j] = self.slab[p][s].data_ptr()
        with torch.cuda.stream(st):
            self.ptr_d.copy_(self.ptr_h, non_blocking=True)
        B.tqfx4_moe_experts(L.ex, L.rt, self.ptr_d, out, ws, st)
        return out, sel_idx, sel_w
