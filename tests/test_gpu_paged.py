"""The paged cache (pages of 64 rows, a device-side free-page stack) against the oracle, its page
accounting, and the decode loop captured in a CUDA graph.

Whole requests run in lockstep with the oracle exactly as for the dense cache (bit-exact rows,
positions and kept sets; outputs and scores within the path's tolerances). The page accounting is
exact: after every call a unit of length n holds the pages of slots [0, n], no page is held twice,
and held plus free pages are the whole pool, turn after turn. A graph replay of the decode loop
gives the same bits as the eager loop."""
import numpy as np
import pytest
import torch

import oracle
from gpu_harness import check_stage1, check_units, gpu_run, make_inputs, oracle_units, sample_units, unit_rows
from paper_2608_08569_gb300 import (DEV_CAPACITY, CacheDesc, allocate_paged_cache, paged_pages_in_use,
                                    voxzip_decode_step_paged, voxzip_get_status)
from paper_2608_08569_gb300 import workloads as W
from paper_2608_08569_gb300.session import Session

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def built():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2608_08569_gb300 import build
    build.build_library()
    oracle.build()
    voxzip_get_status()


def _pages_for(w):
    """A pool that holds stage 1 of every unit plus one page each."""
    return w.units * ((max(w.in_len) + 63) // 64 + 2)


def check_pages(c):
    """Exact accounting of a paged cache: held pages match the lengths, none is held twice, and
    held + free = the pool."""
    tab = c["page_table"].cpu().numpy()
    ln = c["len"].cpu().numpy()
    mp = tab.shape[-1]
    held = tab[tab >= 0]
    assert len(np.unique(held)) == len(held), "a page is held twice"
    need = np.minimum(ln // 64 + 1, mp)
    have = (tab >= 0).sum(-1)
    np.testing.assert_array_equal(have, need)
    for idx in np.ndindex(ln.shape):
        assert np.all(tab[idx][:need[idx]] >= 0) and np.all(tab[idx][need[idx]:] < 0)
    free = c["free_pages"][: int(c["free_count"].item())].cpu().numpy()
    assert len(np.intersect1d(free, held)) == 0
    assert len(free) + len(held) == c["pages"] and len(np.unique(free)) == len(free)


@pytest.mark.parametrize("name,k", [("short", 16), ("long", 8)])
@pytest.mark.parametrize("compaction", ["ordered", "fill"])
def test_whole_path_paged(name, k, compaction):
    w = W.CONFIGS[name]
    pol = dict(pages=_pages_for(w), compaction=compaction)
    inp = make_inputs(w, "cuda")
    sample = sample_units(w, k)
    rec = gpu_run(w, inp, sample, policy=pol)
    check_stage1(w, inp, rec, sample)
    orc = oracle_units(w, inp, sample, policy=pol)
    diverged = check_units(w, rec, orc, sample, policy=pol)
    assert len(diverged) <= max(1, len(sample) // 8), diverged
    check_pages(rec["session"].cache)


def test_pages_follow_the_cache_over_turns():
    """Several requests (turns) on one paged session: after stage 1 the pool holds the stage-1
    rows, after each eviction only the budgets' pages; the footprint stops growing."""
    w = W.scaled(W.CONFIGS["short"], layers=4, name="short_l4")
    desc = CacheDesc(w.batch, w.layers, w.q_heads, w.kv_heads, w.head_dim, (w.capacity + 63) // 64 * 64, w.dtype)
    sess = Session(desc, w.budget, w.gamma, sink=w.sink, recent_frac=w.recent_frac, pages=_pages_for(w))
    inp = make_inputs(w, "cuda")
    sp = inp["spans"]
    i32 = lambda a: torch.as_tensor(np.asarray(a), dtype=torch.int32, device="cuda")
    out = torch.empty(w.layers, w.batch, w.q_heads, w.head_dim, dtype=w.dtype, device="cuda")
    peaks = []
    for turn in range(3):
        sess.prefill(inp["k_pre"], inp["v_pre"], i32(w.in_len), i32([w.audio_begin] * w.batch), i32(w.audio_len),
                     i32(sp.off), i32(sp.start), i32(sp.end), i32(sp.groups))
        check_pages(sess.cache)
        peak = paged_pages_in_use(sess.cache)
        for t in range(1, w.steps + 1):
            sess.decode(inp["q"][t - 1], inp["kn"][t - 1], inp["vn"][t - 1], inp["new_pos"][t - 1], out)
            if t % w.interval == 0:
                sess.evict()
                check_pages(sess.cache)
                units = w.units
                assert paged_pages_in_use(sess.cache) == units * (w.budget[0] // 64 + 1)
            peak = max(peak, paged_pages_in_use(sess.cache))
        peaks.append(peak)
    assert voxzip_get_status() == 0
    assert peaks[0] == peaks[1] == peaks[2]


def test_pool_exhaustion_is_reported_not_fatal():
    """A pool too small for stage 1: the units that did not fit are skipped with
    VOXZIP_DEV_CAPACITY (length 0, no page), the others are fused; decoding the skipped ones
    reports the same bit and leaves them alone."""
    w = W.scaled(W.CONFIGS["short"], layers=2, name="short_l2")
    desc = CacheDesc(w.batch, w.layers, w.q_heads, w.kv_heads, w.head_dim, (w.capacity + 63) // 64 * 64, w.dtype)
    per_unit = (w.in_len[0] // 4) // 64 + 2
    sess = Session(desc, w.budget, w.gamma, pages=w.units * per_unit // 2)
    inp = make_inputs(w, "cuda")
    sp = inp["spans"]
    i32 = lambda a: torch.as_tensor(np.asarray(a), dtype=torch.int32, device="cuda")
    sess.prefill(inp["k_pre"], inp["v_pre"], i32(w.in_len), i32([w.audio_begin] * w.batch), i32(w.audio_len),
                 i32(sp.off), i32(sp.start), i32(sp.end), i32(sp.groups))
    assert voxzip_get_status() & DEV_CAPACITY
    c = sess.cache
    ln = c["len"].cpu().numpy()
    skipped = c["page_table"][..., 0].cpu().numpy() < 0
    assert skipped.any() and (~skipped).any()
    assert np.all(ln[skipped] == 0) and np.all(ln[~skipped] > 0)
    out = torch.empty(w.layers, w.batch, w.q_heads, w.head_dim, dtype=w.dtype, device="cuda")
    sess.decode(inp["q"][0], inp["kn"][0], inp["vn"][0], inp["new_pos"][0], out)
    assert voxzip_get_status() & DEV_CAPACITY
    ln2 = c["len"].cpu().numpy()
    np.testing.assert_array_equal(ln2[skipped], 0)
    np.testing.assert_array_equal(ln2[~skipped], ln[~skipped] + 1)


@pytest.mark.parametrize("paged", [False, True])
def test_decode_loop_graph_replays_the_eager_loop(paged):
    """The decode loop captured once and replayed after a fresh stage 1 gives the eager loop's
    outputs, scores, positions and rows bit for bit."""
    w = W.scaled(W.CONFIGS["short"], layers=6, steps=96, name="short_l6")
    cap = (w.capacity + 63) // 64 * 64
    desc = CacheDesc(w.batch, w.layers, w.q_heads, w.kv_heads, w.head_dim, cap, w.dtype)
    inp = make_inputs(w, "cuda")
    sp = inp["spans"]
    i32 = lambda a: torch.as_tensor(np.asarray(a), dtype=torch.int32, device="cuda")
    args = (inp["k_pre"], inp["v_pre"], i32(w.in_len), i32([w.audio_begin] * w.batch), i32(w.audio_len),
            i32(sp.off), i32(sp.start), i32(sp.end), i32(sp.groups))
    res = []
    for mode in ("eager", "graph"):
        sess = Session(desc, w.budget, w.gamma, pages=_pages_for(w) if paged else None)
        out = torch.zeros(w.steps, w.layers, w.batch, w.q_heads, w.head_dim, dtype=w.dtype, device="cuda")
        sess.prefill(*args)
        if mode == "eager":
            for t in range(1, w.steps + 1):
                sess.decode(inp["q"][t - 1], inp["kn"][t - 1], inp["vn"][t - 1], inp["new_pos"][t - 1], out[t - 1])
                if t % w.interval == 0:
                    sess.evict()
        else:
            # warm the plans eagerly on one request, capture, then replay after a fresh stage 1
            for t in range(1, w.steps + 1):
                sess.decode(inp["q"][t - 1], inp["kn"][t - 1], inp["vn"][t - 1], inp["new_pos"][t - 1], out[t - 1])
                if t % w.interval == 0:
                    sess.evict()
            sess.prefill(*args)
            g = sess.capture_loop(inp["q"][:w.steps], inp["kn"][:w.steps], inp["vn"][:w.steps],
                                  inp["new_pos"][:w.steps], out, w.interval)
            out.zero_()
            sess.prefill(*args)
            g.replay()
        torch.cuda.synchronize()
        assert voxzip_get_status() == 0
        c = sess.cache
        sel = tuple(torch.as_tensor(x, device="cuda") for x in zip(*[(b, l, h) for b in range(w.batch)
                                                                       for l in range(w.layers)
                                                                       for h in range(w.kv_heads)]))
        n = c["len"].clone()
        res.append(dict(out=out.clone(), len=n, score=c["score"].clone(), pos=c["pos"].clone(),
                        k=unit_rows(c, sel, "k", w.head_dim).clone(), v=unit_rows(c, sel, "v", w.head_dim).clone()))
    a, b = res
    assert torch.equal(a["out"], b["out"]) and torch.equal(a["len"], b["len"])
    n = a["len"].flatten()
    for key in ("score", "pos"):
        fa, fb = a[key].flatten(0, 2), b[key].flatten(0, 2)
        for u in range(len(n)):
            assert torch.equal(fa[u, :n[u]], fb[u, :n[u]]), key
    for key in ("k", "v"):
        for u in range(len(n)):
            assert torch.equal(a[key][u, :n[u]], b[key][u, :n[u]]), key
