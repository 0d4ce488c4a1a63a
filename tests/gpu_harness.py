"""Runs a workload through the CUDA path (via the C ABI) and sampled units through the oracle on
the same seeded inputs, and compares them unit by unit.

Tolerances (from the path's arithmetic; the derivation is in the design notes):
  * slot maps, positions, lengths, kept sets: bit-exact;
  * stage-1 cache rows: bit-exact against the oracle's stored rows (both round the fp32 group
    mean once to the cache dtype), and within half a cache-dtype ulp of the exact fp64 mean;
  * attention outputs: 2e-2 absolute for bf16 caches (the output is rounded to bf16 and PV may
    use bf16 probabilities), 1e-4 absolute for fp32 caches;
  * scores (fp32): 1e-4 relative;
  * an eviction may keep a different set only where the oracle's margin between its N-th kept
    and best evicted history score is within the score tolerance; that unit is then no longer
    compared (its cache legitimately differs), and the share of such units is bounded.
"""
from __future__ import annotations

import concurrent.futures as cf
import math
import os

import numpy as np
import torch

import oracle
from paper_2608_08569_gb300 import CacheDesc, voxzip_get_status
from paper_2608_08569_gb300 import workloads as W
from paper_2608_08569_gb300.session import Session

SCORE_RTOL = 1e-4
SCORE_ATOL = 1e-20


def out_tol(w):
    return 2e-2 if w.dtype == torch.bfloat16 else 1e-4


def make_inputs(w, device, steps=None):
    spans = W.make_spans(w)
    k, v = W.make_prefill(w, device)
    q, kn, vn, npos = W.make_steps(w, device, steps=steps)
    return dict(spans=spans, k_pre=k, v_pre=v, q=q, kn=kn, vn=vn, new_pos=npos)


def make_anchors(w, spans, device):
    """Anchor rows [B][L][Hkv][A][D], A = the most anchor rows any sequence needs."""
    A = max(int(spans.groups[spans.off[b]:spans.off[b + 1]].sum()) for b in range(w.batch))
    g = torch.Generator(device=device)
    g.manual_seed(77 + w.seed)
    shape = (w.batch, w.layers, w.kv_heads, max(A, 1), w.head_dim)
    ak = (0.5 * torch.randn(shape, generator=g, device=device)).to(w.dtype)
    av = (0.5 * torch.randn(shape, generator=g, device=device)).to(w.dtype)
    return ak, av


def sample_units(w, k, seed=0):
    """All units when there are at most k, else k spread over sequences, layers and heads."""
    all_units = [(b, l, h) for b in range(w.batch) for l in range(w.layers) for h in range(w.kv_heads)]
    if len(all_units) <= k:
        return all_units
    rng = np.random.default_rng(seed)
    pick = {(0, 0, 0), (w.batch - 1, w.layers - 1, w.kv_heads - 1)}
    while len(pick) < k:
        pick.add(all_units[int(rng.integers(len(all_units)))])
    return sorted(pick)


def unit_budget(w, policy, b, l):
    """The budget of unit (b, l, .): per sequence, or per layer when the policy gives [B][L]."""
    bl = (policy or {}).get("budget_bl")
    return int(bl[b][l]) if bl is not None else int(w.budget[b])


def unit_rows(c, sel, which, D):
    """K or V rows [k][C][D] of the selected units (bi, li, hi): the dense cache, or gathered from a
    paged cache's pool through its page table (slots without a page read pool row 0)."""
    bi, li, hi = sel
    if which in c:
        return c[which][bi, li, hi]
    tab = c["page_table"][bi, li, hi]                       # [k][max_pages]
    C = tab.shape[1] * 64
    slots = torch.arange(C, device=tab.device)
    rows = tab[:, slots // 64].clamp(min=0).long() * 64 + slots % 64
    return c[which + "_pool"].view(-1, D)[rows]


def gpu_run(w, inp, sample, steps=None, anchors=None, policy=None):
    """The whole path on the GPU through the C ABI; records the sampled units. `policy` (optional)
    holds history (bool), compaction ("ordered" / "fill"), budget_bl ([B][L] budgets) and pages
    (a paged cache of that many pages)."""
    S = w.steps if steps is None else steps
    dev = inp["q"].device   # the prefill may be in pinned host memory
    B, L, Hq, H, D, G = w.batch, w.layers, w.q_heads, w.kv_heads, w.head_dim, w.group
    pol = policy or {}
    cap = w.capacity if pol.get("pages") is None else (w.capacity + 63) // 64 * 64   # paged: whole pages
    desc = CacheDesc(B, L, Hq, H, D, cap, w.dtype)
    sess = Session(desc, pol.get("budget_bl", w.budget), w.gamma, sink=w.sink, recent_frac=w.recent_frac,
                   history=pol.get("history", True), compaction=pol.get("compaction", "ordered"), device=dev,
                   pages=pol.get("pages"))
    sp = inp["spans"]
    i32 = lambda a: torch.as_tensor(np.asarray(a), dtype=torch.int32, device=dev)
    slot_map = torch.full((B, w.stride), -1, dtype=torch.int32, device=dev)
    ak, av = anchors if anchors is not None else (None, None)
    voxzip_get_status()  # clear earlier bits
    sess.prefill(inp["k_pre"], inp["v_pre"], i32(w.in_len), i32([w.audio_begin] * B), i32(w.audio_len),
                 i32(sp.off), i32(sp.start), i32(sp.end), i32(sp.groups), slot_map=slot_map, anchor_k=ak,
                 anchor_v=av)
    c = sess.cache
    bi = torch.tensor([u[0] for u in sample], device=dev)
    li = torch.tensor([u[1] for u in sample], device=dev)
    hi = torch.tensor([u[2] for u in sample], device=dev)
    ar = torch.arange(len(sample), device=dev)
    sel = (bi, li, hi)
    rec = dict(stage1_len=c["len"][bi, li, hi].cpu().numpy(), stage1_k=unit_rows(c, sel, "k", D).cpu(),
               stage1_v=unit_rows(c, sel, "v", D).cpu(), stage1_pos=c["pos"][bi, li, hi].cpu().numpy(),
               slot_map=slot_map.cpu().numpy())
    out = torch.empty(L, B, Hq, D, dtype=w.dtype, device=dev)
    outs, sb, lb, kp = [], [], [], []
    maxbud = max(sess.budget_host)
    for t in range(1, S + 1):
        sess.decode(inp["q"][t - 1], inp["kn"][t - 1], inp["vn"][t - 1], inp["new_pos"][t - 1], out)
        outs.append(out[li, bi].view(len(sample), H, G, D)[ar, hi].clone())
        if t % w.interval == 0:
            sb.append(c["score"][bi, li, hi].clone())
            lb.append(c["len"][bi, li, hi].clone())
            sess.evict()
            kp.append(c["pos"][bi, li, hi, :maxbud].clone())
    rec["status"] = voxzip_get_status()
    rec["out"] = torch.stack(outs).float().cpu().numpy() if outs else np.zeros((0, len(sample), G, D))
    rec["score_before"] = torch.stack(sb).cpu().numpy() if sb else None
    rec["len_before"] = torch.stack(lb).cpu().numpy() if lb else None
    rec["kept_pos"] = torch.stack(kp).cpu().numpy() if kp else None
    rec["len"] = c["len"][bi, li, hi].cpu().numpy()
    rec["score"] = c["score"][bi, li, hi].cpu().numpy()
    rec["pos"] = c["pos"][bi, li, hi].cpu().numpy()
    rec["k"] = unit_rows(c, sel, "k", D).cpu()
    rec["v"] = unit_rows(c, sel, "v", D).cpu()
    rec["session"] = sess
    return rec


def _anchor_unit(anchors, w, spans, b, l, h):
    if anchors is None:
        return None, None
    A = int(spans.groups[spans.off[b]:spans.off[b + 1]].sum())
    f = lambda t: t[b, l, h, :A].to("cpu", torch.float64).numpy()
    return f(anchors[0]), f(anchors[1])


def oracle_units(w, inp, sample, steps=None, anchors=None, workers=None, policy=None):
    """run_unit of the oracle for every sampled unit, in parallel threads (ctypes drops the GIL)."""
    S = w.steps if steps is None else steps
    orc = oracle.default()
    args = []
    for (b, l, h) in sample:
        u = W.unit_inputs(w, inp["spans"], inp["k_pre"], inp["v_pre"], inp["q"], inp["kn"], inp["vn"],
                          inp["new_pos"], b, l, h, steps=S)
        ak, av = _anchor_unit(anchors, w, inp["spans"], b, l, h)
        args.append((u, ak, av, b, l))
    pol = policy or {}

    def one(a):
        u, ak, av, b, l = a
        return orc.run_unit(u["xk"], u["xv"], u["in_len"], u["audio_begin"], u["audio_len"], u["span_start"],
                            u["span_end"], u["span_groups"], q=u["q"], k_new=u["k_new"], v_new=u["v_new"],
                            new_pos=u["new_pos"], gamma=w.gamma, scale=1.0 / math.sqrt(w.head_dim),
                            interval=w.interval, budget=unit_budget(w, policy, b, l), sink=w.sink,
                            recent_frac=w.recent_frac, capacity=w.capacity, anchor_k=ak, anchor_v=av,
                            cache_is_bf16=w.dtype == torch.bfloat16, history=pol.get("history", True),
                            fill=pol.get("compaction", "ordered") == "fill")

    with cf.ThreadPoolExecutor(max_workers=workers or os.cpu_count() or 4) as ex:
        return list(ex.map(one, args))


def check_stage1(w, inp, rec, sample, anchors=None):
    """Stage-1 rows, positions, lengths and slot maps against the oracle's stage 1."""
    orc = oracle.default()
    bf16 = w.dtype == torch.bfloat16
    for i, (b, l, h) in enumerate(sample):
        u = W.unit_inputs(w, inp["spans"], inp["k_pre"], inp["v_pre"], inp["q"][:1], inp["kn"][:1],
                          inp["vn"][:1], inp["new_pos"][:1], b, l, h)
        ak, av = _anchor_unit(anchors, w, inp["spans"], b, l, h)
        for x, anc, got in ((u["xk"], ak, rec["stage1_k"]), (u["xv"], av, rec["stage1_v"])):
            r = orc.stage1(x, u["in_len"], u["audio_begin"], u["audio_len"], u["span_start"], u["span_end"],
                           u["span_groups"], anchor=anc, cache_is_bf16=bf16, capacity=w.capacity)
            n = r["n"]
            assert rec["stage1_len"][i] == n, (b, l, h)
            g = got[i, :n].double().numpy()
            np.testing.assert_array_equal(g, r["stored"], err_msg=f"stage-1 rows of unit {(b, l, h)}")
            ulp = np.abs(r["exact"]) * (2.0 ** (-8 if bf16 else -23)) + 1e-6
            assert np.all(np.abs(g - r["exact"]) <= ulp)
            np.testing.assert_array_equal(rec["stage1_pos"][i, :n], r["pos"])
            np.testing.assert_array_equal(rec["slot_map"][b, :u["in_len"]], r["slot_map"])


def _nth_score(scores, n, T, M, N, pos=None):
    """The N-th best history score; the history lies between the sinks and the recent window in
    slot order, or in position order when `pos` is given (hole-filling caches)."""
    mid = scores[T:n - M] if pos is None else scores[np.argsort(pos[:n], kind="stable")][T:n - M]
    cand = np.sort(mid)[::-1]
    return cand[N - 1] if N >= 1 else math.inf


def check_units(w, rec, orc_results, sample, steps=None, policy=None):
    """Lockstep comparison; returns the list of units that legitimately diverged at a near-tie."""
    pol = policy or {}
    S = w.steps if steps is None else steps
    tol = out_tol(w)
    assert rec["status"] == 0, f"device status bits {rec['status']:#x}"
    diverged = []
    stats = dict(max_out_err=0.0, max_score_rel=0.0, evictions=0)
    for i, ((b, l, h), o) in enumerate(zip(sample, orc_results)):
        bud = unit_budget(w, policy, b, l)
        M = math.floor(float(np.float32(w.recent_frac)) * bud) if pol.get("history", True) else bud - w.sink
        N = bud - w.sink - M
        ev = 0
        gone = False
        for t in range(1, S + 1):
            err = np.abs(rec["out"][t - 1, i] - o["out"][t - 1]).max()
            stats["max_out_err"] = max(stats["max_out_err"], float(err))
            assert err <= tol, f"unit {(b, l, h)} step {t}: output error {err:.3g} > {tol}"
            if t % w.interval:
                continue
            n = int(o["len_before"][ev])
            assert rec["len_before"][ev, i] == n, f"unit {(b, l, h)} eviction {ev}: length"
            gs, os_ = rec["score_before"][ev, i, :n], o["score_before"][ev, :n]
            bad = np.abs(gs - os_) > SCORE_RTOL * np.abs(os_) + SCORE_ATOL
            stats["max_score_rel"] = max(stats["max_score_rel"], float(
                (np.abs(gs - os_) / np.maximum(np.abs(os_), 1e-30)).max()))
            stats["evictions"] += 1
            assert not bad.any(), (f"unit {(b, l, h)} eviction {ev}: {bad.sum()} scores off, worst rel "
                                   f"{(np.abs(gs - os_) / np.maximum(np.abs(os_), 1e-30)).max():.3g}")
            m = min(n, bud)
            if not np.array_equal(rec["kept_pos"][ev, i, :m], o["kept_pos"][ev, :m]):
                thr = _nth_score(os_, n, w.sink, M, N,
                                 pos=o["pos_before"][ev] if pol.get("compaction") == "fill" else None)
                assert o["margin"][ev] <= SCORE_RTOL * thr + SCORE_ATOL, (
                    f"unit {(b, l, h)} eviction {ev}: kept sets differ with margin {o['margin'][ev]:.3g} "
                    f"(threshold score {thr:.3g})")
                diverged.append(((b, l, h), t))
                gone = True
                break
            ev += 1
        if gone:
            continue
        n = o["n"]
        assert rec["len"][i] == n
        np.testing.assert_array_equal(rec["pos"][i, :n], o["pos"])
        np.testing.assert_allclose(rec["score"][i, :n], o["score"], rtol=SCORE_RTOL, atol=SCORE_ATOL)
        np.testing.assert_array_equal(rec["k"][i, :n].double().numpy(), o["K"])
        np.testing.assert_array_equal(rec["v"][i, :n].double().numpy(), o["V"])
    check_units.last_stats = stats
    return diverged
