"""Host-side driver of the three C-ABI calls for one batch of sequences.

A ``Session`` owns the device cache (K, V, score, pos, len; or, paged, the page pools, the page
table and the free-page stack), runs stage 1 once per request, then one decode step per
generated token over all layers and an eviction every ``interval`` steps. It keeps a host-side
upper bound on the cache length (read back once after stage 1) so that every decode launch is
sized without a device-to-host sync; the decode loop of a request can therefore be captured once
in a CUDA graph and replayed (``capture_loop``).
"""
from __future__ import annotations

import torch

from . import _native as N


class Session:
    """`budget` holds one budget per sequence, or per sequence and layer ([B][L]); `history` and
    `compaction` select the eviction policy (see voxzip_evict_ex)."""

    def __init__(self, desc: N.CacheDesc, budget, gamma: float, *, sink: int = 4, recent_frac: float = 0.2,
                 history: bool = True, compaction: str = "ordered", device="cuda", cache=None,
                 pages: int | None = None):
        self.desc = desc
        self.device = torch.device(device)
        self.gamma = float(gamma)
        self.sink = int(sink)
        self.recent_frac = float(recent_frac)
        self.history = bool(history)
        self.compaction = compaction
        self.budget = torch.tensor(budget, dtype=torch.int32, device=self.device)
        self.budget_host = [int(b) for b in self.budget.flatten().tolist()]
        self.paged = pages is not None
        if cache is not None:
            self.cache = cache
        elif self.paged:
            self.cache = N.allocate_paged_cache(desc, pages, self.device)
        else:
            self.cache = N.allocate_cache(desc, self.device)
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
        if self.paged:
            N.voxzip_anchor_fuse_paged(self.desc, c, k_prefill, v_prefill, in_len, audio_begin, audio_len, span_off,
                                       span_start, span_end, span_groups, slot_map=slot_map, anchor_k=anchor_k,
                                       anchor_v=anchor_v, workspace=self.workspace, stream=stream)
        else:
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
        if self.paged:
            N.voxzip_decode_step_paged(self.desc, c, layer_begin, lc, q, k_new, v_new, new_pos, self.gamma, out,
                                       max_len=self.n_max + 1, stream=stream)
        else:
            N.voxzip_decode_step(self.desc, layer_begin, lc, q, k_new, v_new, new_pos, c["k"], c["v"], c["score"],
                                 c["pos"], c["len"], self.gamma, out, max_len=self.n_max + 1, stream=stream)
        if layer_begin + lc == self.desc.layers:
            self.n_max += 1

    def evict(self, *, layer_begin=0, layer_count=None, stream=None):
        c = self.cache
        lc = self.desc.layers if layer_count is None else layer_count
        if self.paged:
            N.voxzip_evict_paged(self.desc, c, layer_begin, lc, self.budget, sink=self.sink,
                                 recent_frac=self.recent_frac, history=self.history, compaction=self.compaction,
                                 stream=stream)
        elif self.history and self.compaction == "ordered" and self.budget.dim() == 1:
            N.voxzip_evict(self.desc, layer_begin, lc, c["k"], c["v"], c["score"], c["pos"], c["len"], self.budget,
                           sink=self.sink, recent_frac=self.recent_frac, stream=stream)
        else:
            N.voxzip_evict_ex(self.desc, layer_begin, lc, c["k"], c["v"], c["score"], c["pos"], c["len"],
                              self.budget, sink=self.sink, recent_frac=self.recent_frac, history=self.history,
                              compaction=self.compaction, stream=stream)
        if layer_begin + lc == self.desc.layers:
            self.n_max = min(self.n_max, max(self.budget_host))

    # decode loop in a CUDA graph ---------------------------------------------------------------------
    def capture_loop(self, q, k_new, v_new, new_pos, out, interval: int, *, launch_events=None,
                     segments: bool = False):
        """Captures the decode loop of one request: step t (1-based) decodes with q[t-1], k_new[t-1],
        v_new[t-1], new_pos[t-1] into out[t-1], and evicts when t % interval == 0. Call it right
        after a prefill of the request's shape (it starts from that cache length bound); replaying
        the returned graph after each later prefill of the same shape runs the whole loop with one
        host call. With `launch_events` (a list), timing events (created with external=True) are
        captured too and appended as (kind, start, end, launches): around every decode launch
        ("decode", ..., 1), or with `segments` around each run of decode launches between two
        evictions ("decode", ..., steps in the run: the launches keep overlapping one another as in
        the plain graph), and around every eviction ("evict", ..., 1). The graph records into them
        on every replay, so they must outlive it."""
        n0 = self.n_max
        stream = torch.cuda.Stream(device=self.device)
        stream.wait_stream(torch.cuda.current_stream(self.device))
        graph = torch.cuda.CUDAGraph()
        with torch.cuda.stream(stream):
            with torch.cuda.graph(graph, stream=stream):
                steps = q.shape[0]
                mk = lambda: (torch.cuda.Event(enable_timing=True, external=True),
                              torch.cuda.Event(enable_timing=True, external=True))
                ev, run = None, 0
                for t in range(1, steps + 1):
                    if launch_events is not None and ev is None:
                        ev = mk()
                        ev[0].record()
                    self.decode(q[t - 1], k_new[t - 1], v_new[t - 1], new_pos[t - 1], out[t - 1])
                    run += 1
                    if ev is not None and (not segments or t % interval == 0 or t == steps):
                        ev[1].record()
                        launch_events.append(("decode", ev[0], ev[1], run))
                        ev, run = None, 0
                    if t % interval == 0:
                        eev = None
                        if launch_events is not None:
                            eev = mk()
                            eev[0].record()
                        self.evict()
                        if eev is not None:
                            eev[1].record()
                            launch_events.append(("evict", eev[0], eev[1], 1))
        torch.cuda.current_stream(self.device).wait_stream(stream)
        self.n_max = n0
        return graph
