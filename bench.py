#!/usr/bin/env python
"""Benchmark of the VoxZip KV-compression path on GB300.

One bench step is one request of the workload run through the whole path via the C ABI:
stage-1 fusion of the resident prefilled K/V, then every decode step over all 48 layers
(fused append + GQA attention + decayed-score update) with an eviction every `interval` steps.
The reported value is decode steps per second of the whole job (each decode step advances every
sequence of the batch by one token through all layers), stage 1 and evictions included. By
default each request's decode loop (its decodes and evictions) replays from one CUDA graph
captured once, each launch a programmatic dependent of the one before; stage 1 runs eagerly.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--workload stress] [--impl voxzip|reference]
                  [--loop graph|eager] [--compaction ordered|fill] [--paged]
  python bench.py --part embed [--steps K] [--warmup W]

`--part embed` measures stage 1 where the paper runs it instead: ASR segments of 4 x 60 min of
audio to spans (Eq. 3, on the host) and the fusion of the prompt embeddings (d_model 2048) with the
embedded transcriptions as anchors; one step fuses the four sequences once.

The JSON line also carries the decode, eviction and stage-1 rooflines, the decode and eviction
kernels at the four target points (60-min and 10-min audio, each at the 20x and 4x budgets:
`targets`), the end-to-end rate from pinned host memory (`e2e`) and the oracle's rate on the host
cores (`cpu_baseline`).

Under torchrun each rank runs its own replica of the workload on its own GPU (the units of the
path are independent, so there is no data-path collective); the time is the max over ranks.
`--impl reference` times the fp64 CPU oracle on a bounded sample of the same workload instead.
"""
from __future__ import annotations

import argparse
import concurrent.futures as cf
import json
import math
import os
import statistics
import subprocess
import sys
import tempfile
import time

import numpy as np
import torch

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "decode steps/s + HBM GB/s (% of GB300 peak) for fused attn+score+evict at 4x/20x"
UNIT = "decode steps/s"
FALLBACK_HBM_GBS = 6800.0


def parse_args():
    p = argparse.ArgumentParser(description=__doc__, formatter_class=argparse.RawDescriptionHelpFormatter)
    p.add_argument("--gpus", type=int, default=1)
    p.add_argument("--steps", type=int, default=5)
    p.add_argument("--warmup", type=int, default=3)
    p.add_argument("--impl", choices=["voxzip", "reference"], default="voxzip")
    p.add_argument("--workload", default="stress")
    p.add_argument("--no-e2e", action="store_true")
    p.add_argument("--no-cpu-baseline", action="store_true")
    p.add_argument("--no-targets", action="store_true",
                   help="skip the decode/evict rooflines at the four target points (60-min and 10-min audio "
                        "at the 20x and 4x budgets)")
    p.add_argument("--cpu-units", type=int, default=0, help="units in the oracle sample (0: one per core)")
    p.add_argument("--compaction", choices=["ordered", "fill"], default="ordered",
                   help="eviction compaction: ordered (Eq. 7-8, default) or hole filling")
    p.add_argument("--paged", action="store_true", help="K/V in a paged cache (pages of 64 rows)")
    p.add_argument("--loop", choices=["graph", "eager"], default="graph",
                   help="graph (default): each request's decode loop replays from one captured CUDA graph, "
                        "stage 1 stays eager; eager: one host launch per decode and eviction")
    p.add_argument("--graph", action="store_true", help="same as --loop graph")
    p.add_argument("--part", choices=["path", "embed"], default="path",
                   help="path: the KV-compression path (default); embed: embedding-level stage 1")
    return p.parse_args()


def cores() -> int:
    try:
        return len(os.sched_getaffinity(0))
    except AttributeError:
        return os.cpu_count() or 1


def profiled_traffic_ratio(profile: str, sources) -> float | None:
    """DRAM traffic / algorithmic bytes from a committed ncu summary, or None when the kernel's
    sources changed since that capture (the summary records a hash of them)."""
    import hashlib
    import re
    path = os.path.join(ROOT, "profiles", profile)
    if not os.path.exists(path):
        return None
    text = open(path).read()
    ratio = re.search(r"traffic_ratio: ([0-9.]+)", text)
    digest = re.search(r"source_sha256: ([0-9a-f]+)", text)
    if not ratio or not digest:
        return None
    h = hashlib.sha256()
    for f in sources:
        with open(os.path.join(ROOT, "paper_2608_08569_gb300", "csrc", f), "rb") as fh:
            h.update(fh.read())
    return float(ratio.group(1)) if h.hexdigest()[:len(digest.group(1))] == digest.group(1) else None


def peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(path):
        with open(path) as f:
            d = json.load(f)
        return float(d["hbm_gbs"]), "measured"
    return FALLBACK_HBM_GBS, "fallback"


# ----------------------------------------------------------------------------- distributed

def dist_setup():
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if world > 1:
        import torch.distributed as dist
        backend = "nccl" if torch.cuda.is_available() else "gloo"
        if backend == "nccl":
            torch.cuda.set_device(local)
        dist.init_process_group(backend=backend)
    return rank, world, local


def barrier(world):
    if world > 1:
        import torch.distributed as dist
        dist.barrier()


def max_over_ranks(x: float, world: int) -> float:
    if world == 1:
        return x
    import torch.distributed as dist
    dev = "cuda" if dist.get_backend() == "nccl" else "cpu"
    t = torch.tensor([x], dtype=torch.float64, device=dev)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


# ----------------------------------------------------------------------------- clocks

class ClockSampler:
    """nvidia-smi clock / throttle-reason samples every 200 ms while the timed region runs."""
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, device_index: int):
        self.dev = device_index
        self.proc = None
        self.path = None

    def __enter__(self):
        fd, self.path = tempfile.mkstemp(suffix=".csv")
        os.close(fd)
        sel = []
        try:
            uuid = str(torch.cuda.get_device_properties(self.dev).uuid)
            sel = ["-i", uuid if uuid.startswith("GPU-") else "GPU-" + uuid]
        except Exception:
            sel = []
        try:
            self.f = open(self.path, "w")
            self.proc = subprocess.Popen(["nvidia-smi", *sel, f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits",
                                          "-lms", "200"], stdout=self.f, stderr=subprocess.DEVNULL)
        except OSError:
            self.proc = None
        time.sleep(0.25)
        return self

    def __exit__(self, *exc):
        time.sleep(0.25)
        if self.proc is not None:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()
            self.f.close()

    def summary(self):
        if self.proc is None or not os.path.exists(self.path):
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        rows = []
        with open(self.path) as f:
            for line in f:
                parts = [x.strip() for x in line.split(",")]
                if len(parts) >= 9 and parts[1].replace(".", "").isdigit():
                    rows.append(parts)
        os.unlink(self.path)
        if not rows:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["no samples"]}
        sm = [float(r[1]) for r in rows]
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({n for r in rows for n, v in zip(names, r[5:9]) if v.lower().startswith("active")})
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": float(rows[0][2]), "reasons": reasons,
                "samples": len(rows), "power_w_max": max(float(r[3]) for r in rows if r[3].replace(".", "").isdigit())}


# ----------------------------------------------------------------------------- algorithmic bytes

def decode_bytes(w, n_after):
    """Bytes a decode launch over all layers must move: per unit, every cached K and V row once
    (2 D e bytes per row), each score read and written (8 B), q in and out (2 G D e), k_new and
    v_new in and their append (4 D e), and the new position (4 B)."""
    es = 2 if w.dtype == torch.bfloat16 else 4
    D, G = w.head_dim, w.group
    per_b = [n * (2 * D * es + 8) + (2 * G * D + 4 * D) * es + 4 for n in n_after]
    return w.layers * w.kv_heads * sum(per_b)


def evict_bytes(w, n_before, moved_rows):
    """Bytes an eviction must move (Eq. 7-8): each unit over budget reads its scores and positions
    once for the selection (8 B per slot), and every kept row that changes slot is read and
    written with its K, V, score and position. That is every kept row after the first evicted slot
    for the ordered compaction, and at most n - budget rows for hole filling. moved_rows[u] is
    counted from the positions before and after the eviction."""
    es = 2 if w.dtype == torch.bfloat16 else 4
    row = 2 * w.head_dim * es + 8
    return int(8 * int(n_before.sum()) + 2 * row * int(moved_rows.sum()))


# ----------------------------------------------------------------------------- GPU arm

class Runner:
    """One workload's resident inputs and session. With `share` (a dense Runner of a workload that
    differs only in its budget), the inputs, the cache memory and the outputs are that runner's."""

    def __init__(self, w, device, compaction="ordered", paged=False, share=None):
        from paper_2608_08569_gb300 import CacheDesc
        from paper_2608_08569_gb300 import workloads as W
        from paper_2608_08569_gb300.session import Session
        self.w = w
        self.dev = device
        if share is not None:
            for n in ("spans", "span_args", "k_pre", "v_pre", "q", "kn", "vn", "npos", "out"):
                setattr(self, n, getattr(share, n))
        else:
            self.spans = W.make_spans(w)
            i32 = lambda a: torch.as_tensor(np.asarray(a), dtype=torch.int32, device=device)
            self.span_args = (i32(w.in_len), i32([w.audio_begin] * w.batch), i32(w.audio_len), i32(self.spans.off),
                              i32(self.spans.start), i32(self.spans.end), i32(self.spans.groups))
            self.k_pre, self.v_pre = W.make_prefill(w, device)
            self.q, self.kn, self.vn, self.npos = W.make_steps(w, device)
            self.out = torch.empty(w.steps, w.layers, w.batch, w.q_heads, w.head_dim, dtype=w.dtype, device=device)
        cap = (w.capacity + 63) // 64 * 64 if paged else w.capacity
        self.desc = CacheDesc(w.batch, w.layers, w.q_heads, w.kv_heads, w.head_dim, cap, w.dtype)
        # a paged pool as large as the dense cache: the footprint reported is the pages in use
        self.pages = w.units * (cap // 64) if paged else None
        self.sess = Session(self.desc, w.budget, w.gamma, sink=w.sink, recent_frac=w.recent_frac,
                            compaction=compaction, device=device, pages=self.pages,
                            cache=None if share is None else share.sess.cache)
        self.graph = None

    def capture(self):
        """Captures the decode loop twice after a stage 1: `graph` as it runs (back-to-back launches,
        each a programmatic dependent of the one before), and `graph_timed` with timing events
        around every eviction and around each run of decode launches between two evictions (the
        decode launches of a run still overlap one another), for the rooflines."""
        w, s = self.w, self.sess
        s.prefill(self.k_pre, self.v_pre, *self.span_args[:3], *self.span_args[3:])
        self.graph = s.capture_loop(self.q, self.kn, self.vn, self.npos, self.out, w.interval)
        s.prefill(self.k_pre, self.v_pre, *self.span_args[:3], *self.span_args[3:])
        self.graph_events = []
        self.graph_timed = s.capture_loop(self.q, self.kn, self.vn, self.npos, self.out, w.interval,
                                          launch_events=self.graph_events, segments=True)

    def request_graph(self):
        """One request with the decode loop replayed from the graph."""
        s = self.sess
        s.prefill(self.k_pre, self.v_pre, *self.span_args[:3], *self.span_args[3:])
        self.graph.replay()

    def request(self, timers=None, lengths=None, evict_timers=None, moved=None, pages=None, stage1_timers=None):
        """One request: stage 1, then every decode step with evictions. With `timers` (and
        `evict_timers`), records a CUDA event pair around every decode (evict) launch on the launch
        stream. With `moved`, records per eviction the units' lengths and moved rows (this syncs).
        With `pages` (paged cache), records the pages in use after stage 1 and around the first
        eviction (this syncs)."""
        w, s = self.w, self.sess
        if stage1_timers is not None:
            s0, s1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            s0.record()
        s.prefill(self.k_pre, self.v_pre, *self.span_args[:3], *self.span_args[3:])
        if stage1_timers is not None:
            s1.record()
            stage1_timers.append((s0, s1))
        if pages is not None:
            from paper_2608_08569_gb300 import paged_pages_in_use
            pages.append(paged_pages_in_use(s.cache))
        n = s.cache["len"][:, 0, 0].tolist() if lengths is not None else None
        stream = torch.cuda.current_stream()
        for t in range(1, w.steps + 1):
            if timers is not None:
                e0 = torch.cuda.Event(enable_timing=True)
                e1 = torch.cuda.Event(enable_timing=True)
                e0.record(stream)
            s.decode(self.q[t - 1], self.kn[t - 1], self.vn[t - 1], self.npos[t - 1], self.out[t - 1])
            if timers is not None:
                e1.record(stream)
                timers.append((e0, e1))
            if n is not None:
                n = [x + 1 for x in n]
                lengths.append(("decode", list(n)))
            if t % w.interval == 0:
                if n is not None:
                    lengths.append(("evict", list(n)))
                    n = [min(x, b) for x, b in zip(n, w.budget)]
                if moved is not None:
                    pos_before = s.cache["pos"].clone()
                    n_before = s.cache["len"].clone()
                if evict_timers is not None:
                    f0 = torch.cuda.Event(enable_timing=True)
                    f1 = torch.cuda.Event(enable_timing=True)
                    f0.record(stream)
                if pages is not None and t == w.interval:
                    pages.append(paged_pages_in_use(s.cache))
                s.evict()
                if pages is not None and t == w.interval:
                    pages.append(paged_pages_in_use(s.cache))
                if evict_timers is not None:
                    f1.record(stream)
                    evict_timers.append((f0, f1))
                if moved is not None:
                    moved.append(moved_rows(pos_before, n_before, s.cache["pos"], s.cache["len"]))


def launch_durations(events):
    """Per-launch durations (ms) of decode and eviction launches from an instrumented graph's events:
    a run of decode launches timed as one segment counts its time evenly over its launches."""
    dec, ev = [], []
    for kind, a, b, count in events:
        t = a.elapsed_time(b)
        if kind == "decode":
            dec += [t / count] * count
        else:
            ev.append(t)
    return dec, ev


def moved_rows(pos_before, n_before, pos_after, n_after):
    """(lengths before, rows that changed slot) per unit of one eviction: the slots below the new
    length whose position changed received a row (positions of a unit are unique)."""
    C = pos_before.shape[-1]
    pb = pos_before.reshape(-1, C)
    pa = pos_after.reshape(-1, C)
    nb = n_before.reshape(-1).long()
    na = n_after.reshape(-1).long()
    idx = torch.arange(C, device=pb.device)
    differs = (pb != pa) & (idx[None, :] < na[:, None])
    shrank = na < nb
    moved = torch.where(shrank, differs.sum(1), torch.zeros_like(na))
    return nb[shrank].cpu().numpy(), moved.cpu().numpy()


# ----------------------------------------------------------------------------- target points

# The four target points: the 60-min and 10-min audio workloads, each at the 20x and 4x budgets.
TARGETS = (("60-min 20x", "stress"), ("60-min 4x", "stress_4x"), ("10-min 20x", "long"), ("10-min 4x", "long_4x"))
TARGET_FRAC = 0.70


class _Flush:
    """A read-only pass over 1 GiB (torch's sum): evicts L2 without leaving dirty lines behind."""

    def __init__(self, device):
        self.buf = torch.empty(256 << 20, dtype=torch.float32, device=device)
        self.out = torch.empty((), dtype=torch.float32, device=device)

    def __call__(self):
        torch.sum(self.buf, dim=(0,), out=self.out)


def _graph_replay_ms(body, reps=3):
    """Captures `body` once (after one eager run that sets up plans and tensor maps) and returns the
    replay times in ms (the first replay is a warm-up)."""
    s = torch.cuda.Stream()
    s.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(s):
        body()
    torch.cuda.current_stream().wait_stream(s)
    torch.cuda.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g):
        body()
    out = []
    for r in range(reps + 1):
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record()
        g.replay()
        e1.record()
        torch.cuda.synchronize()
        if r:
            out.append(e0.elapsed_time(e1))
    return out, g


def _steady_cache(w, n, extra, device, seed=7):
    """A dense cache of workload w's shape with every unit at length n: seeded N(0, 1) K and V rows,
    uniform scores, positions in time order (the state the request loop keeps after evictions)."""
    from paper_2608_08569_gb300 import CacheDesc, allocate_cache
    desc = CacheDesc(w.batch, w.layers, w.q_heads, w.kv_heads, w.head_dim, n + extra, w.dtype)
    c = allocate_cache(desc, device)
    g = torch.Generator(device=device)
    g.manual_seed(seed)
    for b in range(w.batch):
        c["k"][b].normal_(generator=g)
        c["v"][b].normal_(generator=g)
    c["score"].uniform_(generator=g)
    c["pos"].copy_(torch.arange(desc.capacity, dtype=torch.int32, device=device).expand_as(c["pos"]))
    c["len"].fill_(n)
    return desc, c


def _frac(nbytes, us, peak):
    gbs = nbytes / us / 1e3
    return {"achieved": round(gbs, 1), "frac": round(gbs / peak, 4), "avg_launch_us": round(us, 2)}


def flushed_decode(w, r, device, peak, flush, NL=8):
    """The decode kernel alone at the workload's mean steady-state length (budget + interval / 2),
    each launch after an L2 flush; median over the launches of two graph replays."""
    from paper_2608_08569_gb300 import voxzip_decode_step, voxzip_get_status
    n = max(w.budget) + w.interval // 2
    desc, c = _steady_cache(w, n, 64, device)
    q, kn, vn, npos, out = r.q[0], r.kn[0], r.vn[0], r.npos[0], r.out[0]
    evs = [(torch.cuda.Event(enable_timing=True, external=True), torch.cuda.Event(enable_timing=True, external=True))
           for _ in range(NL)]

    def body():
        for a, b in evs:
            c["len"].fill_(n)
            flush()
            a.record()
            voxzip_decode_step(desc, 0, w.layers, q, kn, vn, npos, c["k"], c["v"], c["score"], c["pos"], c["len"],
                               w.gamma, out, max_len=n + 1)
            b.record()
    times = []
    _, g = _graph_replay_ms(body, reps=1)
    for _ in range(2):
        g.replay()
        torch.cuda.synchronize()
        times += [a.elapsed_time(b) for a, b in evs]
    if voxzip_get_status() != 0:
        raise RuntimeError("device status word set by the flushed decode")
    us = statistics.median(times) * 1000.0
    res = _frac(decode_bytes(w, [n + 1] * w.batch), us, peak)
    res["n"] = n + 1
    del c, g
    return res


def flushed_evict(w, device, peak, flush, fill=False, NL=6):
    """The eviction kernel alone at the workload's steady state (budget + interval rows per unit,
    uniform scores), each launch after restoring that state and an L2 flush."""
    from paper_2608_08569_gb300 import voxzip_evict, voxzip_evict_ex, voxzip_get_status
    n = max(w.budget) + w.interval
    desc, c = _steady_cache(w, n, 64, device, seed=8)
    ref = {k: v.clone() for k, v in c.items()}
    bud = torch.tensor(w.budget, dtype=torch.int32, device=device)
    evs = [(torch.cuda.Event(enable_timing=True, external=True), torch.cuda.Event(enable_timing=True, external=True))
           for _ in range(NL)]

    def launch():
        if fill:
            voxzip_evict_ex(desc, 0, w.layers, c["k"], c["v"], c["score"], c["pos"], c["len"], bud, sink=w.sink,
                            recent_frac=w.recent_frac, compaction="fill")
        else:
            voxzip_evict(desc, 0, w.layers, c["k"], c["v"], c["score"], c["pos"], c["len"], bud, sink=w.sink,
                         recent_frac=w.recent_frac)

    def body():
        for a, b in evs:
            for k in c:
                c[k].copy_(ref[k])
            flush()
            a.record()
            launch()
            b.record()
    times = []
    _, g = _graph_replay_ms(body, reps=1)
    for _ in range(2):
        g.replay()
        torch.cuda.synchronize()
        times += [a.elapsed_time(b) for a, b in evs]
    for k in c:                       # one more, untimed: the rows that changed slot
        c[k].copy_(ref[k])
    launch()
    torch.cuda.synchronize()
    if voxzip_get_status() != 0:
        raise RuntimeError("device status word set by the flushed eviction")
    nb, mv = moved_rows(ref["pos"], ref["len"], c["pos"], c["len"])
    us = statistics.median(times) * 1000.0
    res = _frac(evict_bytes(w, nb, mv), us, peak)
    res["n_before"] = n
    del c, ref, g
    return res


def decode_loop(w, r, device, peak, NL=32):
    """Back-to-back decode launches from one CUDA graph (each a programmatic dependent of the one
    before, no flush: the cache stays in L2 when it fits, as in a serving loop), against the same
    loop of plain streaming reads of the same bytes (voxzip_stream_read): the most a loop of
    launches of that size reaches. Starts at the budget, as after an eviction."""
    from paper_2608_08569_gb300 import voxzip_decode_step, voxzip_get_status, voxzip_stream_read
    n0 = max(w.budget)
    desc, c = _steady_cache(w, n0, NL + 64, device, seed=9)
    q, kn, vn, npos, out = r.q[0], r.kn[0], r.vn[0], r.npos[0], r.out[0]

    def dec():
        c["len"].fill_(n0)
        for k in range(NL):
            voxzip_decode_step(desc, 0, w.layers, q, kn, vn, npos, c["k"], c["v"], c["score"], c["pos"], c["len"],
                               w.gamma, out, max_len=n0 + k + 1)
    nbytes = sum(decode_bytes(w, [n0 + k + 1] * w.batch) for k in range(NL)) / NL
    nb16 = int(nbytes) // 16 * 16
    buf = torch.empty(nb16 // 4, dtype=torch.int32, device=device).random_(1 << 30)
    sink = torch.zeros(1, dtype=torch.int32, device=device)

    def rd():
        c["len"].fill_(n0)
        for _ in range(NL):
            voxzip_stream_read(buf, nb16, sink)
    t_dec = statistics.median(_graph_replay_ms(dec)[0]) * 1000.0 / NL
    if voxzip_get_status() != 0:
        raise RuntimeError("device status word set by the decode loop")
    t_rd = statistics.median(_graph_replay_ms(rd)[0]) * 1000.0 / NL
    del c, buf
    gbs = nbytes / t_dec / 1e3
    cache_mb = w.units * (n0 + NL) * 4 * w.head_dim / 1e6   # K and V (bf16) the loop streams
    return {"us_per_step": round(t_dec, 2), "gbs": round(gbs, 1), "frac": round(gbs / peak, 4),
            "read_us_per_step": round(t_rd, 2), "read_gbs": round(nbytes / t_rd / 1e3, 1),
            "frac_of_read": round(t_rd / t_dec, 4), "launches": NL, "n_start": n0 + 1,
            "l2_resident": cache_mb < 64.0}


def request_view(r, peak, reps=2):
    """The decode and evict kernels as they run in the workload's request (stage 1, then the decode
    loop replayed from the instrumented CUDA graph: events around every eviction and every run of
    decode launches between two evictions, no flush)."""
    w = r.w
    lengths, moved = [], []
    r.request(lengths=lengths)
    r.request(moved=moved)
    torch.cuda.synchronize()
    r.capture()
    dec_t, ev_t = [], []
    for _ in range(reps):
        r.sess.prefill(r.k_pre, r.v_pre, *r.span_args[:3], *r.span_args[3:])
        r.graph_timed.replay()
        torch.cuda.synchronize()
        d, e = launch_durations(r.graph_events)
        dec_t += d
        ev_t += e
    dec_lens = [n for kind, n in lengths if kind == "decode"]
    dec_bytes = sum(decode_bytes(w, n) for n in dec_lens) * reps
    ev_bytes = sum(evict_bytes(w, nb, mv) for nb, mv in moved) * reps
    dec = _frac(dec_bytes / len(dec_t), 1000.0 * sum(dec_t) / len(dec_t), peak)
    ev = _frac(ev_bytes / max(1, len(ev_t)), 1000.0 * sum(ev_t) / max(1, len(ev_t)), peak)
    r.graph = r.graph_timed = None
    r.graph_events = []
    return dec, ev


def targets_leg(main, device, peak, compaction="ordered", main_request=None):
    """Decode and eviction against the measured HBM peak at the four target points, three ways:
    `request` as the workload's request runs them, `flushed` one launch at a time after an L2 flush
    (the HBM-bound number), `loop` back-to-back launches against a plain read of the same bytes."""
    from paper_2608_08569_gb300 import workloads as W
    flush = _Flush(device)
    runners = {"stress": main}
    res = {}
    for label, name in TARGETS:
        w = W.CONFIGS[name]
        if name == "stress" and main.w.name == "stress":
            r = main
        elif name == "stress_4x" and main.w.name == "stress":
            r = Runner(w, device, compaction=compaction, share=main)
        elif name == "long_4x" and "long" in runners:
            r = Runner(w, device, compaction=compaction, share=runners["long"])
        else:
            r = Runner(w, device, compaction=compaction)
        runners[name] = r
        if r is main and main_request is not None:   # the timed region above measured this one
            keys = ("achieved", "frac", "avg_launch_us")
            dec_req = {k: main_request[0][k] for k in keys}
            ev_req = {k: main_request[1][k] for k in keys} if main_request[1] else None
        else:
            r.request()   # warm-up
            dec_req, ev_req = request_view(r, peak)
        # a cache of at most 64 MB stays in L2 from launch to launch: its rate there is effective
        dec_req["l2_resident"] = w.units * (max(w.budget) + w.interval) * 4 * w.head_dim / 1e6 < 64.0
        res[label] = {
            "workload": name, "budget": max(w.budget),
            "decode": {"request": dec_req, "flushed": flushed_decode(w, r, device, peak, flush),
                       "loop": decode_loop(w, r, device, peak)},
            "evict": {"request": ev_req, "flushed": flushed_evict(w, device, peak, flush,
                                                                  fill=compaction == "fill")},
        }
        torch.cuda.empty_cache()
    del runners
    res["how"] = {
        "request": "the workload's request (stage 1 + every decode step + evictions) replayed from the "
                   "instrumented CUDA graph (events around each eviction and around each run of decode launches "
                   "between two evictions), L2 not flushed (a 10-min cache of 43-203 MB stays partly in L2 "
                   "between launches); algorithmic bytes from the request's lengths and moved rows",
        "flushed": "one launch at a time at the steady state (decode: budget + interval/2 rows per unit; "
                   "evict: budget + interval), a read-only 1 GiB pass before each launch, median of 12-16 "
                   "launches: the HBM-bound number",
        "loop": "32 decode launches back to back from one CUDA graph (programmatic dependent launches, no "
                "flush), as in the request's graph loop but without the per-launch events: frac = algorithmic "
                "bytes / time against the HBM peak (an effective rate where the cache stays in L2, "
                "l2_resident), frac_of_read = the same loop of plain streaming reads of the same bytes "
                "(voxzip_stream_read) / the decode loop",
        "target": f">= {TARGET_FRAC} of the measured HBM peak ({peak} GB/s)"}
    return res


def gpu_arm(args, rank, world, local):
    from paper_2608_08569_gb300 import workloads as W
    w = W.CONFIGS[args.workload]
    dev = torch.device("cuda", local)
    torch.cuda.set_device(dev)
    r = Runner(w, dev, compaction=args.compaction, paged=args.paged)
    for _ in range(args.warmup):
        r.request()
    lengths = []
    if args.graph:
        r.capture()
        r.request(lengths=lengths)   # the lengths of one request (same in every replay)
        r.request_graph()
    torch.cuda.synchronize()
    barrier(world)
    timers, ev_timers, st1_timers = [], [], []
    with ClockSampler(local) as clk:
        torch.cuda.synchronize()
        barrier(world)
        e0 = torch.cuda.Event(enable_timing=True)
        e1 = torch.cuda.Event(enable_timing=True)
        e0.record()
        for k in range(args.steps):
            if args.graph and k < args.steps - 1:
                r.request_graph()
            elif args.graph:  # the last request replays the instrumented copy (events per run of launches)
                s0, s1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
                s0.record()
                r.sess.prefill(r.k_pre, r.v_pre, *r.span_args[:3], *r.span_args[3:])
                s1.record()
                st1_timers.append((s0, s1))
                r.graph_timed.replay()
            else:
                r.request(timers=timers, lengths=lengths if k == 0 else None, evict_timers=ev_timers,
                          stage1_timers=st1_timers)
        e1.record()
        torch.cuda.synchronize()
        barrier(world)
    if args.graph:  # launch times of the instrumented replay, as if every replay took them
        dec_dur, ev_dur = launch_durations(r.graph_events)
        dec_dur, ev_dur = dec_dur * args.steps, ev_dur * args.steps
    else:
        dec_dur = [a.elapsed_time(b) for a, b in timers]
        ev_dur = [a.elapsed_time(b) for a, b in ev_timers]
    ms = e0.elapsed_time(e1)
    ms_max = max_over_ranks(ms, world)
    total_steps = world * args.steps * w.steps
    value = total_steps / (ms_max / 1000.0)

    # Roofline of the dominant kernel (the decode step): algorithmic bytes over event-timed duration.
    dec_lens = [n for kind, n in lengths if kind == "decode"]
    bytes_per_request = sum(decode_bytes(w, n) for n in dec_lens)
    dec_ms = sum(dec_dur)
    launches = len(dec_dur)
    avg_ms = dec_ms / launches
    achieved = bytes_per_request * args.steps / (dec_ms / 1000.0) / 1e9
    peak, peak_kind = peaks()
    n_evict = w.steps // w.interval
    tr = profiled_traffic_ratio("decode_mma_kernel_stress.md", ["decode_mma.cu", "ptx.cuh", "common.cuh"])
    alg_per_launch = bytes_per_request / max(1, len(dec_lens))
    roofline = {"bound": "hbm", "achieved": round(achieved, 1), "peak": peak, "unit": "GB/s",
                "frac": round(achieved / peak, 4),
                "traffic": None if tr is None or w.name != "stress" else int(tr * alg_per_launch),
                "kernel": "decode_mma_kernel (append + GQA attention + decayed score)",
                "traffic_source": "profiles/decode_mma_kernel_stress.md: dram bytes / algorithmic bytes on steady "
                                  "launches, times this run's algorithmic bytes per launch",
                "peak_source": f"{peak_kind} hbm_gbs",
                "avg_launch_us": round(avg_ms * 1000.0, 2),
                "alg_bytes_per_launch": int(bytes_per_request / max(1, len(dec_lens))),
                "decode_share_of_step": round(dec_ms / ms, 4)}
    # The same split at the first eviction: before it the cache holds the whole stage-1 output.
    pre = [i for i in range(len(dec_dur)) if i % w.steps < w.interval]
    post = [i for i in range(len(dec_dur)) if i % w.steps >= w.interval]
    for name, ids in (("before_first_evict", pre), ("after_first_evict", post)):
        b = sum(decode_bytes(w, dec_lens[i % w.steps]) for i in ids)
        t = sum(dec_dur[i] for i in ids)
        if t > 0:
            roofline[f"achieved_{name}"] = round(b / (t / 1000.0) / 1e9, 1)
    # kernels per request: 3 stage-1 kernels (5 paged), one decode launch per step, one evict per interval
    gpu_launches = args.steps * ((5 if args.paged else 3) + w.steps + n_evict)

    # The eviction kernel against the same peak: bytes from an untimed replay of one request.
    moved, pages = [], ([] if args.paged else None)
    r.request(moved=moved, pages=pages)
    torch.cuda.synchronize()
    ev_bytes = sum(evict_bytes(w, nb, mv) for nb, mv in moved)
    ev_ms = sum(ev_dur)
    if ev_dur and ev_ms > 0:
        ev_ach = ev_bytes * args.steps / (ev_ms / 1000.0) / 1e9
        etr = profiled_traffic_ratio("evict_kernel_stress.md", ["evict.cu", "common.cuh"]) \
            if args.compaction == "ordered" else None
        roofline_evict = {"bound": "hbm", "achieved": round(ev_ach, 1), "peak": peak, "unit": "GB/s",
                          "frac": round(ev_ach / peak, 4),
                          "traffic": None if etr is None or w.name != "stress" else
                          int(etr * ev_bytes / max(1, len(moved))),
                          "kernel": "evict_kernel (top-N select + ordered in-place compaction)"
                          if args.compaction == "ordered" else
                          "evict_fill_kernel (top-N select + hole-filling compaction)",
                          "avg_launch_us": round(1000.0 * ev_ms / len(ev_dur), 2),
                          "alg_bytes_per_launch": int(ev_bytes / max(1, len(moved))),
                          "evict_share_of_step": round(ev_ms / ms, 4)}
    else:
        roofline_evict = None

    # Stage 1 (span scan, slot map and the fusion kernel, timed together): the prefilled K and V read
    # once, the stage-1 rows written with their score and position.
    roofline_stage1 = None
    if st1_timers and dec_lens:
        es = 2 if w.dtype == torch.bfloat16 else 4
        n1 = [x - 1 for x in dec_lens[0]]
        st1_bytes = w.layers * w.kv_heads * sum(2 * il * w.head_dim * es + nn * (2 * w.head_dim * es + 8)
                                                for il, nn in zip(w.in_len, n1))
        st1_ms = sum(a.elapsed_time(b) for a, b in st1_timers) / len(st1_timers)
        per_req_ms = ms / args.steps
        roofline_stage1 = {"bound": "hbm", "achieved": round(st1_bytes / (st1_ms / 1000.0) / 1e9, 1), "peak": peak,
                           "unit": "GB/s", "frac": round(st1_bytes / (st1_ms / 1000.0) / 1e9 / peak, 4),
                           "kernel": "stage 1: span_scan + slot_map + fuse_rows_kernel (timed together)",
                           "avg_call_us": round(st1_ms * 1000.0, 1), "alg_bytes_per_call": int(st1_bytes),
                           "stage1_share_of_step": round(st1_ms / per_req_ms, 4)}

    e2e = None
    if not args.no_e2e:
        e2e = e2e_leg(r, args)
    clocks = clk.summary()
    targets = None
    if not args.no_targets and not args.paged and w.name == "stress":
        with ClockSampler(local) as tclk:
            targets = targets_leg(r, dev, peak, compaction=args.compaction,
                                  main_request=(roofline, roofline_evict))
        targets["clocks"] = tclk.summary()
    result = {
        "metric": METRIC, "value": round(value, 2), "unit": UNIT, "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": round(ms_max / args.steps, 3), "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "bf16" if w.dtype == torch.bfloat16 else "f32",
        "data": "synthetic (seeded; Qwen3-Omni-thinker-shaped K/V/q, ASR-like spans)",
        "config": {"workload": f"{w.name}: {w.description}", "batch": w.batch, "layers": w.layers,
                   "q_heads": w.q_heads, "kv_heads": w.kv_heads, "head_dim": w.head_dim,
                   "prompt_tokens": list(sorted(set(w.in_len))), "budget": list(sorted(set(w.budget))),
                   "gamma": w.gamma, "decode_steps_per_request": w.steps, "evict_interval": w.interval,
                   "compaction": args.compaction, "graph": bool(args.graph),
                   "loop": "graph" if args.graph else "eager",
                   "roofline_timing": ("CUDA events in the last timed request, which replays an instrumented "
                                       "copy of the graph: around every eviction, and around each run of 32 "
                                       "decode launches between two evictions (the decode launches of a run "
                                       "overlap one another as in the plain graph); a run's time counts evenly "
                                       "over its launches")
                                      if args.graph else
                                      "CUDA events around every launch inside the timed region",
                   "paged": None if not args.paged else {
                       "page_rows": 64, "pool_pages": r.pages,
                       "bytes_per_page": 2 * 64 * w.head_dim * (2 if w.dtype == torch.bfloat16 else 4),
                       "pages_after_stage1": pages[0], "pages_before_first_evict": pages[1],
                       "pages_after_first_evict": pages[2],
                       "dense_cache_bytes": w.units * r.desc.capacity * 2 * w.head_dim *
                                            (2 if w.dtype == torch.bfloat16 else 4)},
                   "parallelism": f"replicas x{world} (independent units, no collective)",
                   "l2": "inputs larger than L2 (decode reads ~0.9-7 GB per launch, L2 is 129 MB)"},
        "roofline": roofline, "roofline_evict": roofline_evict, "roofline_stage1": roofline_stage1,
        "gpu_launches": gpu_launches, "clocks": clocks,
        "e2e": e2e, "targets": targets,
    }
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        result["cpu_baseline"] = cpu_sample(w, args.cpu_units, compaction=args.compaction)
    return result


def e2e_leg(r, args):
    """The same metric with every request's inputs taken from pinned host memory and its attention
    outputs copied back. The prompt's prefilled K/V (18.1 GB of the 20.1 GB a 60-min request
    brings) are read by stage 1 itself, straight from pinned host memory over the host link (the
    device addresses page-locked memory directly on GB300's C2C link), so they never take an HBM copy
    that the decode loop, which saturates HBM, would starve. Every step's q / k_new / v_new /
    position and the spans are copied by the copy engines. Two request slots, each with its own
    cache, step buffers and captured decode loop, alternate: while request k decodes in one, request
    k + 1's inputs arrive and its stage 1 runs in the other (prep stream), and request k - 1's
    outputs leave (download stream); events order every reuse."""
    from paper_2608_08569_gb300.session import Session
    w = r.w
    if args.paged or not args.graph:
        return {"value": None, "unit": UNIT, "skipped": "the end-to-end leg runs the dense cache's graph loop"}
    nbytes = lambda t: t.numel() * t.element_size()
    steps_in = ("q", "kn", "vn", "npos")
    need = nbytes(r.k_pre) + nbytes(r.v_pre) + sum(nbytes(getattr(r, n)) for n in steps_in) + nbytes(r.out)
    avail = host_mem_available()
    if avail is not None and avail < 1.5 * need + (8 << 30):
        return {"value": None, "unit": UNIT, "skipped": f"host memory: {avail >> 30} GiB available, "
                                                        f"{need >> 30} GiB of pinned buffers needed"}

    def pin(t):
        h = torch.empty(t.shape, dtype=t.dtype, pin_memory=True)
        h.copy_(t)
        return h
    host_pre = (pin(r.k_pre), pin(r.v_pre))
    host_in = {n: pin(getattr(r, n)) for n in steps_in}
    host_spans = [pin(t) for t in r.span_args]
    h_out = torch.empty(r.out.shape, dtype=r.out.dtype).pin_memory()
    slots = []
    for _ in range(2):
        sess = Session(r.desc, w.budget, w.gamma, sink=w.sink, recent_frac=w.recent_frac,
                       compaction=r.sess.compaction, device=r.dev)
        bufs = {n: torch.empty_like(getattr(r, n)) for n in steps_in + ("out",)}
        for n in steps_in:
            bufs[n].copy_(host_in[n])
        spans = tuple(t.clone() for t in r.span_args)
        # stage 1 once with the length read back, then the request's decode loop captured from there
        sess.prefill(host_pre[0], host_pre[1], *spans[:3], *spans[3:])
        graph = sess.capture_loop(bufs["q"], bufs["kn"], bufs["vn"], bufs["npos"], bufs["out"], w.interval)
        slots.append({"sess": sess, "bufs": bufs, "spans": spans, "graph": graph})
    torch.cuda.synchronize()
    prep_s, down = torch.cuda.Stream(), torch.cuda.Stream()
    comp = torch.cuda.current_stream()
    prepped = [torch.cuda.Event(), torch.cuda.Event()]
    computed = [torch.cuda.Event(), torch.cuda.Event()]
    drained = [torch.cuda.Event(), torch.cuda.Event()]

    def prep(i, first_use):
        sl = slots[i]
        with torch.cuda.stream(prep_s):
            if not first_use:
                prep_s.wait_event(computed[i])   # the slot's previous request is done with it
            for n in steps_in:
                sl["bufs"][n].copy_(host_in[n], non_blocking=True)
            for d, h in zip(sl["spans"], host_spans):
                d.copy_(h, non_blocking=True)
            sl["sess"].prefill(host_pre[0], host_pre[1], *sl["spans"][:3], *sl["spans"][3:], stream=prep_s,
                               read_back=False)
            prepped[i].record(prep_s)

    def compute(i, first_use):
        comp.wait_event(prepped[i])
        if not first_use:
            comp.wait_event(drained[i])          # its previous outputs have left
        slots[i]["graph"].replay()
        computed[i].record(comp)

    def store(i):
        with torch.cuda.stream(down):
            down.wait_event(computed[i])
            h_out.copy_(slots[i]["bufs"]["out"], non_blocking=True)
            drained[i].record(down)

    def run(n_req):
        prep(0, True)
        for k in range(n_req):
            if k + 1 < n_req:
                prep((k + 1) % 2, k + 1 < 2)
            compute(k % 2, k < 2)
            store(k % 2)
        comp.wait_stream(down)
        comp.wait_stream(prep_s)

    run(2)
    torch.cuda.synchronize()
    e0 = torch.cuda.Event(enable_timing=True)
    e1 = torch.cuda.Event(enable_timing=True)
    e0.record()
    run(args.steps)
    e1.record()
    torch.cuda.synchronize()
    ms = e0.elapsed_time(e1)
    from paper_2608_08569_gb300 import voxzip_get_status
    if voxzip_get_status() != 0:
        raise RuntimeError("device status word set in the end-to-end leg")
    pre_bytes = sum(nbytes(t) for t in host_pre)
    copied = sum(nbytes(t) for t in host_in.values()) + sum(nbytes(t) for t in host_spans)
    del slots
    torch.cuda.empty_cache()
    return {"value": round(args.steps * w.steps / (ms / 1000.0), 2), "unit": UNIT,
            "h2d_bytes_per_step": pre_bytes + copied, "d2h_bytes_per_step": nbytes(h_out),
            "h2d_read_by_stage1_bytes": pre_bytes, "h2d_copied_bytes": copied, "ms_per_step": round(ms / args.steps, 3),
            "copies": "prefill K/V streamed from pinned host memory by stage 1 over the host link; step inputs "
                      "copied by the copy engines; two request slots: request k+1's inputs and stage 1 overlap "
                      "request k's decode loop, request k-1's outputs leave meanwhile"}


def host_mem_available():
    try:
        with open("/proc/meminfo") as f:
            for line in f:
                if line.startswith("MemAvailable:"):
                    avail = int(line.split()[1]) * 1024
                    break
            else:
                return None
    except OSError:
        return None
    for path in ("/sys/fs/cgroup/memory.max",):
        try:
            with open(path) as f:
                lim = f.read().strip()
            if lim != "max":
                avail = min(avail, int(lim))
        except (OSError, ValueError):
            pass
    return avail


# ----------------------------------------------------------------------------- oracle (CPU) arm

def sample_units(w, k):
    rng = np.random.default_rng(123)
    all_units = [(b, l, h) for b in range(w.batch) for l in range(w.layers) for h in range(w.kv_heads)]
    idx = rng.choice(len(all_units), size=min(k, len(all_units)), replace=False)
    return [all_units[i] for i in sorted(idx)]


def cpu_sample(w, n_units=0, inputs=None, compaction="ordered"):
    """Times the oracle on a bounded sample: `n_units` units (one per thread), each through the
    whole request; the whole-workload time is the sample's wall time x units / sampled units."""
    import oracle
    from paper_2608_08569_gb300 import workloads as W
    threads = cores()
    n_units = n_units or min(threads, w.units)
    units = sample_units(w, n_units)
    spans = W.make_spans(w)
    if inputs is None:
        inputs = [W.unit_inputs_cpu(w, spans, b, l, h) for (b, l, h) in units]
    orc = oracle.default()

    def one(a):
        u, b = a
        return orc.run_unit(u["xk"], u["xv"], u["in_len"], u["audio_begin"], u["audio_len"], u["span_start"],
                            u["span_end"], u["span_groups"], q=u["q"], k_new=u["k_new"], v_new=u["v_new"],
                            new_pos=u["new_pos"], gamma=w.gamma, scale=1.0 / math.sqrt(w.head_dim),
                            interval=w.interval, budget=w.budget[b], sink=w.sink, recent_frac=w.recent_frac,
                            capacity=w.capacity, cache_is_bf16=w.dtype == torch.bfloat16, fill=compaction == "fill")

    args = [(u, b) for u, (b, l, h) in zip(inputs, units)]
    used = min(threads, len(args))
    t0 = time.perf_counter()
    with cf.ThreadPoolExecutor(max_workers=used) as ex:
        list(ex.map(one, args))
    wall = time.perf_counter() - t0
    full = wall * w.units / len(units)
    t1 = time.perf_counter()
    one(args[0])                      # one unit alone: the single-thread rate
    one_unit = time.perf_counter() - t1
    return {"value": round(w.steps / full, 4), "unit": UNIT, "cores": used, "kind": "oracle",
            "sample": (f"{len(units)} of {w.units} units (seeded choice), each through the whole request "
                       f"({w.steps} decode steps, evictions every {w.interval}); {wall:.1f} s wall on {used} "
                       f"threads, scaled by {w.units}/{len(units)} to the whole workload"),
            "sample_wall_s": round(wall, 2),
            "single_thread_value": round(w.steps / (one_unit * w.units), 5),
            "single_thread_sample": f"one unit alone, {one_unit:.1f} s, scaled by {w.units} units"}, inputs


def reference_arm(args, rank, world):
    from paper_2608_08569_gb300 import workloads as W
    w = W.CONFIGS[args.workload]
    if rank != 0:
        return None
    inputs = None
    for _ in range(args.warmup):
        _, inputs = cpu_sample(w, args.cpu_units, inputs, args.compaction)
    vals, last = [], None
    t0 = time.perf_counter()
    for _ in range(args.steps):
        last, inputs = cpu_sample(w, args.cpu_units, inputs, args.compaction)
        vals.append(last["value"])
    wall = time.perf_counter() - t0
    value = statistics.mean(vals)
    cb = dict(last)
    cb["value"] = round(value, 4)
    return {"metric": METRIC, "value": round(value, 4), "unit": UNIT, "n_gpus": world, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": round(1000.0 * wall / args.steps, 1), "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f64", "impl": "reference",
            "data": "synthetic (seeded; Qwen3-Omni-thinker-shaped K/V/q, ASR-like spans)",
            "config": {"workload": f"{w.name}: {w.description}"}, "cpu_baseline": cb,
            "e2e": {"value": round(value, 4), "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}


# ----------------------------------------------------------------------------- embedding-level stage 1

EMBED_METRIC = "stage-1 embedding fusion (Sec. 3.2.1, Eq. 3-5): sequences/s, 4 x 60 min audio, d_model 2048"


class EmbedRunner:
    """Resident inputs of embedding-level stage 1: prompt embeddings, spans from the ASR
    segments (the library's Eq. 3 helper), and the kept segments' text embeddings."""

    def __init__(self, w, device):
        from paper_2608_08569_gb300 import EmbedDesc, voxzip_segments_to_spans
        from paper_2608_08569_gb300 import workloads as W
        self.w, self.dev = w, device
        self.segs = W.make_segments(w)
        self.e_in = W.make_embeddings(w, device)
        self.text_all = W.make_text_embeddings(w, self.segs, device)
        self.spans_host()
        off, st, en, gr = self.spans
        i32 = lambda x: torch.as_tensor(np.asarray(x), dtype=torch.int32, device=device)
        self.args = [i32(w.in_len), i32([w.audio_begin] * w.batch), i32(w.audio_len), i32(off), i32(st), i32(en),
                     i32(gr)]
        rows = []
        for b, s in enumerate(self.segs):
            first = np.concatenate([[0], np.cumsum(s.text_len)])
            sel = [np.arange(first[i], first[i + 1]) for i in self.seg_index[b]]
            rows.append(np.concatenate(sel) if sel else np.zeros(0, np.int64))
        self.e_text = torch.zeros(w.batch, max(1, max(len(r) for r in rows)), w.d_model, dtype=w.dtype, device=device)
        for b, r in enumerate(rows):
            if len(r):
                self.e_text[b, :len(r)] = self.text_all[b, torch.as_tensor(r, device=device)]
        self.desc = EmbedDesc(w.batch, w.d_model, w.capacity, w.dtype)
        self.out = torch.empty(w.batch, w.capacity, w.d_model, dtype=w.dtype, device=device)
        self.pos = torch.empty(w.batch, w.capacity, dtype=torch.int32, device=device)
        self.len = torch.empty(w.batch, dtype=torch.int32, device=device)

    def spans_host(self):
        """The semantic set of every sequence from its ASR segments (host, Eq. 3)."""
        from paper_2608_08569_gb300 import voxzip_segments_to_spans
        w = self.w
        off, st, en, gr, self.seg_index = [0], [], [], [], []
        for b, s in enumerate(self.segs):
            r = voxzip_segments_to_spans(s.t_start, s.t_end, s.confidence, s.text_len, s.tau_total, w.audio_len[b],
                                         w.audio_begin)
            st += list(r["start"]); en += list(r["end"]); gr += list(r["groups"])
            self.seg_index.append(r["seg_index"])
            off.append(len(st))
        self.spans = (off, st, en, gr)

    def step(self):
        from paper_2608_08569_gb300 import voxzip_embed_fuse
        voxzip_embed_fuse(self.desc, self.e_in, *self.args, self.out, self.pos, self.len, e_text=self.e_text)

    def alg_bytes(self):
        """Embedding rows read (prompt, and one text row per emitted group), fused rows written,
        and the per-row integers (position; source range and anchor row written and read)."""
        w, e = self.w, (2 if self.w.dtype == torch.bfloat16 else 4)
        off, st, en, gr = self.spans
        groups = sum(min(g, b - a) for a, b, g in zip(st, en, gr))
        n_out = int(self.len.sum())
        return (sum(w.in_len) + groups + n_out) * w.d_model * e + n_out * 28 + len(st) * 12


def embed_arm(args, rank, world, local):
    from paper_2608_08569_gb300 import voxzip_get_status
    from paper_2608_08569_gb300 import workloads as W
    w = W.EMBED_CONFIGS["embed_stress"]
    dev = torch.device("cuda", local)
    torch.cuda.set_device(dev)
    r = EmbedRunner(w, dev)
    for _ in range(args.warmup):
        r.step()
    torch.cuda.synchronize()
    if voxzip_get_status() != 0:
        raise RuntimeError("device status word set by embedding-level stage 1")
    barrier(world)
    evs = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(args.steps)]
    with ClockSampler(local) as clk:
        torch.cuda.synchronize()
        barrier(world)
        e0 = torch.cuda.Event(enable_timing=True)
        e1 = torch.cuda.Event(enable_timing=True)
        e0.record()
        for a, b in evs:
            a.record()
            r.step()
            b.record()
        e1.record()
        torch.cuda.synchronize()
        barrier(world)
    ms = e0.elapsed_time(e1)
    ms_max = max_over_ranks(ms, world)
    value = world * args.steps * w.batch / (ms_max / 1000.0)
    launch_ms = sum(a.elapsed_time(b) for a, b in evs) / args.steps
    alg = r.alg_bytes()
    peak, peak_kind = peaks()
    achieved = alg / (launch_ms / 1000.0) / 1e9
    roofline = {"bound": "hbm", "achieved": round(achieved, 1), "peak": peak, "unit": "GB/s",
                "frac": round(achieved / peak, 4), "traffic": None,
                "kernel": "embedding stage 1 (span_scan + slot_map + fuse_wide_kernel, timed together)",
                "peak_source": f"{peak_kind} hbm_gbs", "avg_call_us": round(launch_ms * 1000.0, 2),
                "alg_bytes_per_call": int(alg)}
    e2e = None if args.no_e2e else embed_e2e(r, args)
    clocks = clk.summary()
    result = {
        "metric": EMBED_METRIC, "value": round(value, 2), "unit": "sequences/s", "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": round(ms_max / args.steps, 3),
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
        "dtype": "bf16" if w.dtype == torch.bfloat16 else "f32",
        "data": "synthetic (seeded; N(0,1) embeddings, ASR-like timed segments at 12.5 audio tokens/s)",
        "config": {"workload": f"{w.name}: {w.description}", "batch": w.batch, "d_model": w.d_model,
                   "prompt_tokens": list(sorted(set(w.in_len))), "spans": len(r.spans[1]),
                   "output_rows": int(r.len.sum()), "parallelism": f"replicas x{world}",
                   "l2": "inputs larger than L2 (0.75 GB of embeddings read per step, L2 is 129 MB)"},
        "roofline": roofline, "gpu_launches": 3 * args.steps, "clocks": clocks, "e2e": e2e,
    }
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        result["cpu_baseline"] = embed_cpu_sample(r)
    return result


def embed_e2e(r, args):
    """The same with every step's embeddings and text rows copied from pinned host memory, the
    spans recomputed from the ASR segments on the host (Eq. 3) and copied, and the fused rows
    copied back."""
    nbytes = lambda t: t.numel() * t.element_size()
    h_in = torch.empty(r.e_in.shape, dtype=r.e_in.dtype, pin_memory=True)
    h_in.copy_(r.e_in)
    h_text = torch.empty(r.e_text.shape, dtype=r.e_text.dtype, pin_memory=True)
    h_text.copy_(r.e_text)
    h_out = torch.empty(r.out.shape, dtype=r.out.dtype, pin_memory=True)
    span_bytes = [0]

    def step():
        r.spans_host()
        off, st, en, gr = r.spans
        hs = [torch.as_tensor(np.asarray(x), dtype=torch.int32).pin_memory() for x in (off, st, en, gr)]
        for src, dst in zip(hs, r.args[3:]):
            dst.copy_(src, non_blocking=True)
        span_bytes[0] = sum(nbytes(t) for t in hs)
        r.e_in.copy_(h_in, non_blocking=True)
        r.e_text.copy_(h_text, non_blocking=True)
        r.step()
        h_out.copy_(r.out, non_blocking=True)

    step()
    torch.cuda.synchronize()
    e0 = torch.cuda.Event(enable_timing=True)
    e1 = torch.cuda.Event(enable_timing=True)
    e0.record()
    for _ in range(args.steps):
        step()
    e1.record()
    torch.cuda.synchronize()
    ms = e0.elapsed_time(e1)
    return {"value": round(args.steps * r.w.batch / (ms / 1000.0), 2), "unit": "sequences/s",
            "h2d_bytes_per_step": nbytes(h_in) + nbytes(h_text) + span_bytes[0],
            "d2h_bytes_per_step": nbytes(h_out), "ms_per_step": round(ms / args.steps, 3)}


def embed_cpu_sample(r, cols=16):
    """The oracle's stage 1 on `cols` of the d_model columns of every sequence (stage 1 acts on
    each column alone), one sequence per thread; scaled to whole sequences per second."""
    import oracle
    w = r.w
    oracle.build()
    off, st, en, gr = r.spans
    sel = torch.arange(0, w.d_model, w.d_model // cols, device=r.e_in.device)[:cols]
    xs = [r.e_in[b, :w.in_len[b]][:, sel].double().cpu().numpy() for b in range(w.batch)]
    ts = [r.e_text[b][:, sel].double().cpu().numpy() for b in range(w.batch)]

    def one(b):
        s0, s1 = off[b], off[b + 1]
        oracle.stage1(xs[b], w.in_len[b], w.audio_begin, w.audio_len[b], st[s0:s1], en[s0:s1], gr[s0:s1],
                      anchor=ts[b], cache_is_bf16=True, capacity=w.capacity)

    threads = min(cores(), w.batch)
    t0 = time.perf_counter()
    with cf.ThreadPoolExecutor(threads) as ex:
        list(ex.map(one, range(w.batch)))
    sec = time.perf_counter() - t0
    per_seq = sec / w.batch * threads * (w.d_model / cols)
    return {"value": round(threads / per_seq, 4), "unit": "sequences/s", "cores": threads, "kind": "oracle",
            "sample": f"{cols} of {w.d_model} columns of each of the {w.batch} sequences (all rows), one thread "
                      f"per sequence; scaled by d_model / {cols}"}


def main():
    args = parse_args()
    args.graph = args.graph or args.loop == "graph"
    rank, world, local = dist_setup()
    if args.part == "embed" and args.impl != "reference":
        res = embed_arm(args, rank, world, local)
        if rank == 0:
            print(json.dumps(res), flush=True)
        if world > 1:
            import torch.distributed as dist
            dist.destroy_process_group()
        return
    if args.impl == "reference":
        res = reference_arm(args, rank, world)
    else:
        res = gpu_arm(args, rank, world, local)
        if isinstance(res.get("cpu_baseline"), tuple):
            res["cpu_baseline"] = res["cpu_baseline"][0]
    if rank == 0 and res is not None:
        print(json.dumps(res), flush=True)
    if world > 1:
        import torch.distributed as dist
        dist.destroy_process_group()


if __name__ == "__main__":
    main()
