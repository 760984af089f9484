"""One pass of the hot path for a workload, through the C ABI.

A step processes the nodes of one launch (one pipeline round, Eq. 6, or one
serial node, Eq. 5):
  1. context selection for every node (sva_select_context, Eq. 2-3) and the
     (chunk, level) -> slot lookups;
  2. for pipelined workloads, the availability check (sva_check_pipeline,
     Eq. 7);
  3. the fused 3D-RoPE + cache scatter of the nodes' new K/V and in-place Q
     rotation (sva_rope_kv_write), which also makes this round's states
     readable by the progressive nodes of the same round (Section 3.3);
  4. the batched policy-indexed attention (sva_attend_nodes, Eq. 4; with a
     block-sparse workload sva_attend_nodes_sparse and the workload's seeded
     key-tile mask).
Steps 3 and 4 are stream-ordered kernels; 1 and 2 are host integer work.
"""
from __future__ import annotations

import math

import torch

from . import sva
from .inputs import Inputs, Workload, tile_mask


def geometry_for(w: Workload, spare_slots: int = 2) -> sva.sva_geometry:
    return sva.make_geometry(w.H, w.d, w.F, w.Hp, w.Wp, num_slots=len(w.states) + spare_slots,
                             pairs=w.pairs, max_frames=w.max_frames, theta=w.theta)


class Step:
    def __init__(self, w: Workload, device: str = "cuda", spare_slots: int = 2,
                 workspace: bool = True):
        self.w = w
        self.device = torch.device(device)
        self.policy = sva.POLICIES[w.policy]
        self.cache = sva.Cache(geometry_for(w, spare_slots), device=self.device)
        if workspace:
            ws = torch.empty(self.cache.workspace_bytes(), dtype=torch.uint8, device=self.device)
            self.cache.set_workspace(ws)
        self.own = {}
        self.scale = 1.0 / math.sqrt(w.d)
        self.mask = tile_mask(w).to(self.device) if w.sparse is not None else None

    def prefill(self, inp: Inputs, stream=None):
        """Binds and writes the workload's history states (untimed set-up)."""
        w = self.w
        self.norm = None
        if w.qknorm:
            self.norm = (inp.gamma_k.to(self.device), inp.gamma_q.to(self.device), inp.norm_eps)
        pre = list(w.prefilled)
        for start in range(0, len(pre), sva.MAX_NODES):
            group = pre[start:start + sva.MAX_NODES]
            entries = []
            for (s, c, l) in group:
                slot = self.cache.bind(s, c, l)
                entries.append(dict(seq=s, chunk=c, level=l, own_slot=slot))
            k = torch.stack([inp.history[tuple(st)][0] for st in group]).to(self.device)
            v = torch.stack([inp.history[tuple(st)][1] for st in group]).to(self.device)
            if self.norm is not None:
                self.cache.rope_kv_write_qknorm(entries, k, v, None, self.norm[0], None,
                                                self.norm[2], stream=stream)
            else:
                self.cache.rope_kv_write(entries, k, v, None, stream=stream)
        for st in w.nodes:
            self.own[tuple(st)] = self.cache.bind(*st)

    def node_table(self):
        """Steps 1-2: the node descriptors of this launch (host integer work)."""
        w = self.w
        entries = []
        for (s, b, j) in w.nodes:
            sel = sva.select_context(self.policy, w.K, w.W, b, j)
            if w.round is not None:
                st = sva.check_pipeline(w.K, j, b, sel)
                if st != sva.OK:
                    raise sva.SvaError(st, sva.last_error())
            ctx = [self.cache.lookup(s, c, l) for (c, l) in sel]
            entries.append(dict(seq=s, chunk=b, level=j, own_slot=self.own[(s, b, j)], ctx=ctx,
                                within=sva.WITHIN[w.within]))
        return sva.make_nodes(entries), len(entries)

    def run(self, q, k_new, v_new, out, lse=None, stream=None, rotate_q: bool = True):
        """One pass of the hot path on device tensors [n][T][H][d] (q rotated in place)."""
        nodes, n = self.node_table()
        if self.norm is not None:
            self.cache.rope_kv_write_qknorm(nodes, k_new, v_new, q if rotate_q else None,
                                            self.norm[0], self.norm[1], self.norm[2],
                                            stream=stream)
        else:
            self.cache.rope_kv_write(nodes, k_new, v_new, q if rotate_q else None, stream=stream,
                                     check=False)
        self.attend(nodes, q, out, lse, stream=stream)
        return n

    def attend(self, nodes, q, out, lse=None, stream=None):
        """Step 4 alone (dense or block-sparse, as the workload says)."""
        if self.mask is not None:
            self.cache.attend_nodes_sparse(nodes, q, out, self.mask, lse, self.scale, stream=stream,
                                           check=False)
        else:
            self.cache.attend_nodes(nodes, q, out, lse, self.scale, stream=stream, check=False)

    def device_inputs(self, inp: Inputs):
        d = self.device
        return inp.q.to(d).contiguous(), inp.k_new.to(d).contiguous(), inp.v_new.to(d).contiguous()

    def outputs(self):
        w = self.w
        out = torch.empty((w.n_nodes, w.T, w.H, w.d), dtype=torch.bfloat16, device=self.device)
        lse = torch.empty((w.n_nodes, w.H, w.T), dtype=torch.float32, device=self.device)
        return out, lse

    def close(self):
        self.cache.close()
