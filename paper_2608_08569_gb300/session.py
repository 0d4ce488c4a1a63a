"""Host-side driver of the three C-ABI calls for one batch of sequences.

A ``Session`` owns the device cache (K, V, score, pos, len), runs stage 1 once per request, then
one decode step per generated token over all layers and an eviction every ``interval`` steps.
It keeps a host-side upper bound on the cache length (read back once after stage 1) so that
every decode launch is sized without a device-to-host sync.
"""
from __future__ import annotations

import torch

from . import _native as N


class Session:
    """`budget` holds one budget per sequence, or per sequence and layer ([B][L]); `history` and
    `compaction` select the eviction policy (see voxzip_evict_ex)."""

    def __init__(self, desc: N.CacheDesc, budget, gamma: float, *, sink: int = 4, recent_frac: float = 0.2,
                 history: bool = True, compaction: str = "ordered", device="cuda", cache=None):
        self.desc = desc
        self.device = torch.device(device)
        self.gamma = float(gamma)
        self.sink = int(sink)
        self.recent_frac = float(recent_frac)
        self.history = bool(history)
        self.compaction = compaction
        self.budget = torch.tensor(budget, dtype=torch.int32, device=self.device)
        self.budget_host = [int(b) for b in self.budget.flatten().tolist()]
        self.cache = cache if cache is not None else N.allocate_cache(desc, self.device)
        self.n_max = 0
        self.workspace = None

    # stage 1 -------------------------------------------------------------------------------------
    def prefill(self, k_prefill, v_prefill, in_len, audio_begin, audio_len, span_off, span_start, span_end,
                span_groups, *, anchor_k=None, anchor_v=None, slot_map=None, stream=None, read_back=True):
        """Stage-1 fusion of the prefilled cache (all device tensors, see voxzip_anchor_fuse)."""
        c = self.cache
        need = N.voxzip_anchor_fuse_workspace_size(self.desc, k_prefill.shape[3], span_start.numel())
        if self.workspace is None or self.workspace.numel() < need:
            self.workspace = torch.empty(max(need, 256), dtype=torch.uint8, device=self.device)
        N.voxzip_anchor_fuse(self.desc, k_prefill, v_prefill, in_len, audio_begin, audio_len, span_off,
                             span_start, span_end, span_groups, c["k"], c["v"], c["score"], c["pos"], c["len"],
                             slot_map=slot_map, anchor_k=anchor_k, anchor_v=anchor_v, workspace=self.workspace,
                             stream=stream)
        if read_back:
            self.n_max = int(c["len"].max().item())
        else:
            self.n_max = int(k_prefill.shape[3])  # stage 1 never lengthens a prompt

    # stage 2 -------------------------------------------------------------------------------------
    def decode(self, q, k_new, v_new, new_pos, out, *, layer_begin=0, layer_count=None, stream=None):
        """One decode step for a layer range (all layers by default)."""
        c = self.cache
        lc = self.desc.layers if layer_count is None else layer_count
        N.voxzip_decode_step(self.desc, layer_begin, lc, q, k_new, v_new, new_pos, c["k"], c["v"], c["score"],
                             c["pos"], c["len"], self.gamma, out, max_len=self.n_max + 1, stream=stream)
        if layer_begin + lc == self.desc.layers:
            self.n_max += 1

    def evict(self, *, layer_begin=0, layer_count=None, stream=None):
        c = self.cache
        lc = self.desc.layers if layer_count is None else layer_count
        if self.history and self.compaction == "ordered" and self.budget.dim() == 1:
            N.voxzip_evict(self.desc, layer_begin, lc, c["k"], c["v"], c["score"], c["pos"], c["len"], self.budget,
                           sink=self.sink, recent_frac=self.recent_frac, stream=stream)
        else:
            N.voxzip_evict_ex(self.desc, layer_begin, lc, c["k"], c["v"], c["score"], c["pos"], c["len"],
                              self.budget, sink=self.sink, recent_frac=self.recent_frac, history=self.history,
                              compaction=self.compaction, stream=stream)
        if layer_begin + lc == self.desc.layers:
            self.n_max = min(self.n_max, max(self.budget_host))
