"""Pins that tie the fp64 oracle to what the paper and the mathematics fix.

Each ``pin_*`` takes an ``oracle.Oracle`` and raises AssertionError (or OracleError) when the
oracle disagrees with a hand-worked fixture (``tests/golden``), a closed form, an invariant, a
library routine for a special case, or brute force on a tiny input. ``test_oracle_pins`` runs
them on the committed oracle; ``test_oracle_mutations`` runs them on copies of the oracle with
planted mistakes and expects each mistake to be caught.
"""
from __future__ import annotations

import itertools
import json
import math
import os

import numpy as np
import torch

import oracle as O

GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden")


def _golden(name):
    with open(os.path.join(GOLDEN, name)) as f:
        return json.load(f)


def _num(v):
    if isinstance(v, str):
        named = {"inf": math.inf, "sqrt(2)*ln(3)": math.sqrt(2.0) * math.log(3.0),
                 "1/sqrt(2)": 1.0 / math.sqrt(2.0)}
        if v in named:
            return named[v]
        a, b = v.split("/")
        return float(a) / float(b)
    return float(v)


def _rows(rows):
    return np.array([[_num(v) for v in r] for r in rows])


def _bf16(a):
    """Round to bf16 (torch's RNE cast) and widen back to float64."""
    return torch.from_numpy(np.asarray(a, np.float32)).to(torch.bfloat16).double().numpy()


# ----------------------------------------------------------------------------- stage 1

def pin_stage1_hand(orc):
    """Hand-worked stage-1 example: Eq. 4 means, anchor add, Eq. 5 order, slot map, positions."""
    g = _golden("stage1_hand.json")
    x = np.array([[t, t * t] for t in range(g["in_len"])], float)
    r = orc.stage1(x, g["in_len"], g["audio_begin"], g["audio_len"], g["span_start"], g["span_end"],
                   g["span_groups"])
    assert r["n"] == len(g["expected_rows"])
    np.testing.assert_allclose(r["exact"], _rows(g["expected_rows"]), rtol=0, atol=1e-12)
    np.testing.assert_array_equal(r["pos"], g["expected_pos"])
    np.testing.assert_array_equal(r["slot_map"], g["expected_slot_map"])
    n_anchor = sum(g["span_groups"])
    anchor = np.array([[100.0 * (k + 1), -(k + 1.0)] for k in range(n_anchor)])
    r = orc.stage1(x, g["in_len"], g["audio_begin"], g["audio_len"], g["span_start"], g["span_end"],
                   g["span_groups"], anchor=anchor)
    np.testing.assert_allclose(r["exact"], _rows(g["expected_rows_with_anchor"]), rtol=0, atol=1e-12)
    np.testing.assert_allclose(r["stored"], _rows(g["expected_rows_with_anchor"]), rtol=1e-6, atol=0)

    m = g["more_groups_than_tokens"]
    x = np.array([[t, t * t] for t in range(m["in_len"])], float)
    r = orc.stage1(x, m["in_len"], m["audio_begin"], m["audio_len"], m["span_start"], m["span_end"],
                   m["span_groups"])
    np.testing.assert_allclose(r["exact"], _rows(m["expected_rows"]), rtol=0, atol=1e-12)
    np.testing.assert_array_equal(r["pos"], m["expected_pos"])
    anchor = np.array([[100.0 * (k + 1), -(k + 1.0)] for k in range(sum(m["span_groups"]))])
    r = orc.stage1(x, m["in_len"], m["audio_begin"], m["audio_len"], m["span_start"], m["span_end"],
                   m["span_groups"], anchor=anchor)
    np.testing.assert_allclose(r["exact"], _rows(m["expected_rows_with_anchor"]), rtol=0, atol=1e-12)


def pin_run_unit_fuses_k_and_v_with_their_own_anchors(orc):
    """A whole unit (stage 1, then one decode step, no eviction) fuses K with the K anchors and V
    with the V anchors. With V's rows twice K's (the hand-worked stage-1 example) and V's anchors the
    negated K anchors, the example's means M and anchored means A give, row by row, K = A and
    V = 2M - (A - M) = 3M - A (Eq. 4 and the anchor addition are linear in the rows)."""
    g = _golden("stage1_hand.json")
    x = np.array([[t, t * t] for t in range(g["in_len"])], float)
    anchor = np.array([[100.0 * (k + 1), -(k + 1.0)] for k in range(sum(g["span_groups"]))])
    M, A = _rows(g["expected_rows"]), _rows(g["expected_rows_with_anchor"])
    n1, D = len(M), 2
    cap = n1 + 4
    r = orc.run_unit(x, 2.0 * x, g["in_len"], g["audio_begin"], g["audio_len"], g["span_start"], g["span_end"],
                     g["span_groups"], q=np.zeros((1, 1, D)), k_new=np.zeros((1, D)), v_new=np.zeros((1, D)),
                     new_pos=[1000], gamma=0.9, scale=1.0, interval=1000, budget=cap, capacity=cap,
                     anchor_k=anchor, anchor_v=-anchor)
    assert r["stage1_len"] == n1 and r["n"] == n1 + 1
    np.testing.assert_allclose(r["K"][:n1], A, rtol=1e-6, atol=1e-6)
    np.testing.assert_allclose(r["V"][:n1], 3.0 * M - A, rtol=1e-6, atol=1e-5)


def pin_stage1_fp32_accumulation(orc):
    """Hand-worked IEEE cases for the stored group mean: an fp32 sum in token order (not the exact
    mean rounded once), and the anchor added in fp32 before the one rounding to bf16."""
    for c in _golden("stage1_fp32_accumulation.json")["cases"]:
        rows = np.array(c["rows"], float)[:, None].repeat(2, axis=1)
        n = len(rows)
        anchor = None if c["anchor"] is None else np.full((1, 2), float(c["anchor"]))
        r = orc.stage1(rows, n, 0, n, [0], [n], [1], anchor=anchor, cache_is_bf16=c["cache"] == "bf16")
        assert r["n"] == 1
        assert r["stored"][0, 0] == c["stored"], (c, r["stored"][0, 0])


def pin_stage1_bf16_rounding(orc):
    """Hand-worked round-to-nearest-even of fp32 group means into a bf16 cache."""
    for c in _golden("stage1_bf16_rounding.json")["cases"]:
        rows = np.array(c["rows"], float)[:, None].repeat(2, axis=1)
        n = len(rows)
        r = orc.stage1(rows, n, 0, n, [0], [n], [1], cache_is_bf16=True)
        assert r["n"] == 1
        assert r["stored"][0, 0] == c["stored"], (c, r["stored"][0, 0])
        if not isinstance(c["mean"], str):
            assert r["exact"][0, 0] == c["mean"]


def _random_spans(rng, audio_begin, audio_len, max_len=9, p_gap=0.3, max_groups=3):
    starts, ends, groups = [], [], []
    t = audio_begin
    while t < audio_begin + audio_len:
        if rng.random() < p_gap:
            t += int(rng.integers(1, 4))
            continue
        ln = int(rng.integers(0, max_len + 1))
        e = min(t + ln, audio_begin + audio_len)
        starts.append(t)
        ends.append(e)
        groups.append(int(rng.integers(1, max_groups + 1)))
        t = e
    return starts, ends, groups


def pin_stage1_identity(orc):
    """Spans of length 1, or with n_groups equal to their length, make stage 1 the identity."""
    rng = np.random.default_rng(1)
    D, in_len, ab, al = 16, 60, 7, 40
    x = _bf16(rng.standard_normal((in_len, D)))
    for mode in ("len1", "ng_eq_len"):
        if mode == "len1":
            ss = list(range(ab, ab + al))
            se = [s + 1 for s in ss]
            sg = [int(rng.integers(1, 4)) for _ in ss]
        else:
            ss, se, _ = _random_spans(rng, ab, al)
            sg = [max(1, e - s) for s, e in zip(ss, se)]
        r = orc.stage1(x, in_len, ab, al, ss, se, sg, cache_is_bf16=True)
        assert r["n"] == in_len
        assert np.array_equal(r["stored"], x) and np.array_equal(r["exact"], x)
        np.testing.assert_array_equal(r["slot_map"], np.arange(in_len))
        np.testing.assert_array_equal(r["pos"], np.arange(in_len))


def pin_stage1_structure(orc):
    """Output length, group sizes, slot map and positions follow Eq. 4-5 on random spans; a span
    of identical rows fuses to that row; group sizes sum to the span length and differ by <= 1."""
    rng = np.random.default_rng(2)
    for trial in range(20):
        D = 8
        in_len = int(rng.integers(1, 80))
        ab = int(rng.integers(0, in_len))
        al = int(rng.integers(0, in_len - ab + 1))
        ss, se, sg = _random_spans(rng, ab, al)
        x = _bf16(rng.standard_normal((in_len, D)))
        r = orc.stage1(x, in_len, ab, al, ss, se, sg, cache_is_bf16=True)
        covered = sum(e - s for s, e in zip(ss, se))
        expect_len = (in_len - covered) + sum(min(g, e - s) for s, e, g in zip(ss, se, sg))
        assert r["n"] == expect_len
        sm = r["slot_map"]
        assert sm[0] == 0 and np.all(np.diff(sm) >= 0) and np.all(np.diff(sm) <= 1)
        assert sm[-1] == r["n"] - 1
        # Each slot's position is the first token mapped to it.
        first = np.searchsorted(sm, np.arange(r["n"]), side="left")
        np.testing.assert_array_equal(r["pos"], first)
        for s, e, g in zip(ss, se, sg):
            if e == s:
                continue
            sizes = np.bincount(sm[s:e] - sm[s])
            assert len(sizes) == min(g, e - s) and sizes.sum() == e - s
            assert sizes.max() - sizes.min() <= 1 and np.all(np.diff(sizes) >= 0)
            # The span sum is preserved: sum over groups of |G| * mean.
            np.testing.assert_allclose((sizes[:, None] * r["exact"][sm[s]:sm[s] + len(sizes)]).sum(0),
                                       x[s:e].sum(0), rtol=1e-12, atol=1e-12)
        # Tokens outside every span are copied unchanged.
        inside = np.zeros(in_len, bool)
        for s, e in zip(ss, se):
            inside[s:e] = True
        for t in np.nonzero(~inside)[0]:
            assert np.array_equal(r["stored"][sm[t]], x[t])
        # Stored bf16 values are the exact mean rounded (within half a bf16 ulp + fp32 sum error).
        tol = np.abs(r["exact"]) * (2.0 ** -8) * 1.01 + 1e-6
        assert np.all(np.abs(r["stored"] - r["exact"]) <= tol)
    # A span of identical rows fuses to that row.
    row = _bf16(rng.standard_normal(8))
    x = np.tile(row, (10, 1))
    r = orc.stage1(x, 10, 0, 10, [0], [10], [1], cache_is_bf16=True)
    assert r["n"] == 1 and np.array_equal(r["stored"][0], row)
    np.testing.assert_allclose(r["exact"][0], row, rtol=1e-15)


def pin_stage1_partial_hand(orc):
    """Hand-worked "Partial" stage 1: the same example with the background audio dropped."""
    g = _golden("stage1_hand.json")
    x = np.array([[t, t * t] for t in range(g["in_len"])], float)
    r = orc.stage1(x, g["in_len"], g["audio_begin"], g["audio_len"], g["span_start"], g["span_end"],
                   g["span_groups"], keep_background=False)
    p = g["partial"]
    assert r["n"] == len(p["expected_rows"])
    np.testing.assert_allclose(r["exact"], _rows(p["expected_rows"]), rtol=0, atol=1e-12)
    np.testing.assert_array_equal(r["pos"], p["expected_pos"])
    np.testing.assert_array_equal(r["slot_map"], p["expected_slot_map"])


def pin_stage1_partial_relation(orc):
    """Dropping the background removes exactly the background rows of the full stage 1 and
    nothing else: the remaining rows, positions and their order are the full result's."""
    rng = np.random.default_rng(5)
    for trial in range(20):
        in_len = int(rng.integers(1, 80))
        ab = int(rng.integers(0, in_len))
        al = int(rng.integers(0, in_len - ab + 1))
        ss, se, sg = _random_spans(rng, ab, al)
        x = _bf16(rng.standard_normal((in_len, 4)))
        anchor = _bf16(rng.standard_normal((max(1, sum(sg)), 4)))
        full = orc.stage1(x, in_len, ab, al, ss, se, sg, anchor=anchor, cache_is_bf16=True)
        part = orc.stage1(x, in_len, ab, al, ss, se, sg, anchor=anchor, cache_is_bf16=True,
                          keep_background=False)
        inside = np.zeros(in_len, bool)
        for s, e in zip(ss, se):
            inside[s:e] = True
        background = np.zeros(in_len, bool)
        background[ab:ab + al] = ~inside[ab:ab + al]
        keep_slots = np.unique(full["slot_map"][~background])
        assert part["n"] == len(keep_slots) == full["n"] - int(background.sum())
        np.testing.assert_array_equal(part["stored"], full["stored"][keep_slots])
        np.testing.assert_array_equal(part["exact"], full["exact"][keep_slots])
        np.testing.assert_array_equal(part["pos"], full["pos"][keep_slots])
        assert np.all(part["slot_map"][background] == -1)
        remap = np.full(full["n"], -1)
        remap[keep_slots] = np.arange(len(keep_slots))
        np.testing.assert_array_equal(part["slot_map"][~background], remap[full["slot_map"][~background]])


def pin_segments_hand(orc):
    """Hand-worked confidence filter and Eq. 3 time-to-index map."""
    g = _golden("eq3_segments.json")
    r = orc.segments_to_spans(g["t_start"], g["t_end"], g["confidence"], g["text_len"], g["tau_total"],
                              g["La"], g["audio_begin"], g["threshold"])
    np.testing.assert_array_equal(r["start"], g["expected_start"])
    np.testing.assert_array_equal(r["end"], g["expected_end"])
    np.testing.assert_array_equal(r["groups"], g["expected_groups"])
    np.testing.assert_array_equal(r["seg_index"], g["expected_seg_index"])
    e = g["boundary"]  # exact token boundaries, where the order of Eq. 3's operations shows
    r = orc.segments_to_spans(e["t_start"], e["t_end"], e["confidence"], e["text_len"], e["tau_total"],
                              e["La"], e["audio_begin"], e["threshold"])
    np.testing.assert_array_equal(r["start"], e["expected_start"])
    np.testing.assert_array_equal(r["end"], e["expected_end"])
    e = g["nested"]  # a segment inside the previous one: clipped to an empty span that keeps its text rows
    r = orc.segments_to_spans(e["t_start"], e["t_end"], e["confidence"], e["text_len"], e["tau_total"],
                              e["La"], e["audio_begin"], e["threshold"])
    for k in ("start", "end", "groups", "seg_index"):
        np.testing.assert_array_equal(r[k], e["expected_" + k], err_msg=k)


def pin_segments_properties(orc):
    """On random ASR output the spans are sorted, disjoint, inside the audio region; exactly the
    segments above the threshold are kept, with their text lengths; where segments neither
    overlap nor leave the audio, an interval's length is the number of token boundaries
    k / L_a * tau_total (k integer) its times enclose, counted by brute force."""
    rng = np.random.default_rng(6)
    for trial in range(30):
        La = int(rng.integers(1, 400))
        tau = float(rng.uniform(1.0, 100.0))
        n = int(rng.integers(0, 12))
        cuts = np.sort(rng.uniform(0.0, tau, 2 * n))
        ts, te = cuts[0::2], cuts[1::2]
        conf = rng.uniform(0.0, 1.0, n)
        tl = rng.integers(1, 6, n)
        ab = int(rng.integers(0, 50))
        r = orc.segments_to_spans(ts, te, conf, tl, tau, La, ab, 0.3)
        kept = np.nonzero(conf > 0.3)[0]
        np.testing.assert_array_equal(r["seg_index"], kept)
        np.testing.assert_array_equal(r["groups"], tl[kept])
        st, en = r["start"], r["end"]
        assert np.all(st >= ab) and np.all(en <= ab + La) and np.all(en >= st)
        assert np.all(st[1:] >= en[:-1])
        for k, i in enumerate(kept):
            # Token k' starts at time k' * tau / La; idx(t) = number of token starts in (0, t].
            bounds = np.arange(1, La + 1) * (tau / La)
            lo = int(np.sum(bounds <= ts[i] * (1 + 1e-12)))
            hi = int(np.sum(bounds <= te[i] * (1 + 1e-12)))
            near = lambda t: np.min(np.abs(bounds - t)) < 1e-9 * tau
            if not (near(ts[i]) or near(te[i])):
                assert st[k] - ab == lo and en[k] - ab == hi, (trial, i, st[k] - ab, lo, en[k] - ab, hi)
    # Overlapping or unsorted input: overlaps are clipped, unsorted input is rejected.
    r = orc.segments_to_spans([0.0, 0.5], [1.0, 2.0], [1.0, 1.0], [1, 1], 2.0, 20)
    np.testing.assert_array_equal(r["start"], [0, 10]) and np.testing.assert_array_equal(r["end"], [10, 20])
    for args in (([1.0, 0.5], [2.0, 2.0], [1.0, 1.0], [1, 1], 2.0, 20),   # unsorted
                 ([0.0], [1.0], [1.0], [0], 2.0, 20),                       # no text tokens
                 ([0.0], [1.0], [1.0], [1], 0.0, 20),                       # zero duration
                 ([1.0], [0.5], [1.0], [1], 2.0, 20)):                      # ends before it starts
        try:
            orc.segments_to_spans(*args)
        except O.OracleError:
            continue
        raise AssertionError(f"accepted {args}")


def pin_stage1_errors(orc):
    """Malformed semantic sets are rejected; the output must fit the capacity."""
    x = np.zeros((10, 4))
    bad = [([3, 2], [5, 4], [1, 1]),    # unsorted
           ([2, 3], [5, 6], [1, 1]),    # overlapping
           ([0], [3], [1]),             # starts before the audio region
           ([2], [9], [1]),             # ends after it
           ([2], [4], [0]),             # zero groups
           ([4], [3], [1])]             # end < start
    for ss, se, sg in bad:
        try:
            orc.stage1(x, 10, 1, 7, ss, se, sg)
        except O.OracleError as e:
            assert e.code == O.EINVAL
        else:
            raise AssertionError(f"accepted {ss, se, sg}")
    try:
        orc.stage1(x, 10, 1, 7, [2], [4], [1], capacity=8)
    except O.OracleError as e:
        assert e.code == O.ECAPACITY
    else:
        raise AssertionError("capacity overflow accepted")
    r = orc.stage1(x, 10, 1, 7, [2], [4], [1], capacity=9)
    assert r["n"] == 9


# ----------------------------------------------------------------------------- decode

def pin_decode_hand(orc):
    """Hand-worked decode step with two query heads (Eq. 1, Eq. 2, Eq. 6)."""
    g = _golden("decode_hand.json")
    c = O.UnitCache.from_rows(4, np.array(g["cache_K"], float), np.array(g["cache_V"], float),
                              g["cache_pos"], g["cache_score"])
    out = orc.decode_step(c, _rows(g["q"]), np.array(g["k_new"], float), np.array(g["v_new"], float),
                          g["new_pos"], g["gamma"], _num(g["scale"]))
    np.testing.assert_allclose(out, np.array(g["expected_out"]), rtol=0, atol=1e-12)
    assert c.n == g["expected_n"]
    np.testing.assert_allclose(c.score[:c.n], g["expected_score"], rtol=0, atol=1e-12)
    np.testing.assert_array_equal(c.pos[:c.n], g["expected_pos"])
    np.testing.assert_array_equal(c.K[1], g["k_new"])
    np.testing.assert_array_equal(c.V[1], g["v_new"])


def _random_cache(rng, n, D, cap):
    K = rng.standard_normal((n, D))
    V = rng.standard_normal((n, D))
    return O.UnitCache.from_rows(cap, K, V, np.arange(n))


def pin_decode_full_attention(orc):
    """gamma = 1 without eviction: each output is textbook softmax attention over the whole cache
    (torch's scaled_dot_product_attention, GQA-expanded) and each score is the plain cumulative
    attention mass (H2O accumulation), computed from torch's softmax."""
    rng = np.random.default_rng(3)
    D, G, n0, steps = 32, 4, 9, 6
    c = _random_cache(rng, n0, D, n0 + steps)
    Kall = c.K[:n0].copy()
    Vall = c.V[:n0].copy()
    cum = np.zeros(n0 + steps)
    for t in range(steps):
        q = rng.standard_normal((G, D)) * 2.0
        kn, vn = rng.standard_normal(D), rng.standard_normal(D)
        out = orc.decode_step(c, q, kn, vn, 1000 + t, 1.0, 1.0 / math.sqrt(D))
        Kall = np.vstack([Kall, kn])
        Vall = np.vstack([Vall, vn])
        qt = torch.from_numpy(q)[None, :, None, :]                     # [1, G, 1, D]
        kt = torch.from_numpy(Kall)[None, None].expand(1, G, -1, -1)   # [1, G, n, D]
        vt = torch.from_numpy(Vall)[None, None].expand(1, G, -1, -1)
        ref = torch.nn.functional.scaled_dot_product_attention(qt, kt, vt)[0, :, 0].numpy()
        np.testing.assert_allclose(out, ref, rtol=1e-10, atol=1e-12)
        w = torch.softmax(torch.from_numpy(q) @ torch.from_numpy(Kall).T / math.sqrt(D), dim=-1)
        cum[:len(Kall)] += w.sum(0).numpy()
        np.testing.assert_allclose(c.score[:c.n], cum[:c.n], rtol=1e-12, atol=1e-14)
    np.testing.assert_array_equal(c.pos[n0:c.n], 1000 + np.arange(steps))
    # A caller-chosen softmax scale (the C ABI's sm_scale) replaces 1/sqrt(D): SDPA with that scale.
    c = _random_cache(rng, n0, D, n0 + 1)
    q = rng.standard_normal((G, D))
    kn, vn = rng.standard_normal(D), rng.standard_normal(D)
    out = orc.decode_step(c, q, kn, vn, 2000, 1.0, 0.3)
    kt = torch.from_numpy(c.K[:c.n].copy())[None, None].expand(1, G, -1, -1)
    vt = torch.from_numpy(c.V[:c.n].copy())[None, None].expand(1, G, -1, -1)
    ref = torch.nn.functional.scaled_dot_product_attention(torch.from_numpy(q)[None, :, None, :], kt, vt,
                                                           scale=0.3)[0, :, 0].numpy()
    np.testing.assert_allclose(out, ref, rtol=1e-10, atol=1e-12)


def pin_decode_total_mass(orc):
    """Each softmax sums to 1, so between evictions sum_j A_j(t) = gamma * sum_j A_j(t-1) + G;
    from zero: G (1 - gamma^t) / (1 - gamma)."""
    rng = np.random.default_rng(4)
    D, G, n0 = 16, 3, 5
    for gamma in (0.95, 0.5, 0.999):
        c = _random_cache(rng, n0, D, n0 + 40)
        for t in range(1, 41):
            orc.decode_step(c, rng.standard_normal((G, D)) * 3, rng.standard_normal(D),
                            rng.standard_normal(D), t, gamma, 1 / math.sqrt(D))
            closed = G * (1 - gamma ** t) / (1 - gamma)
            assert abs(c.score[:c.n].sum() - closed) <= 1e-12 * closed, (gamma, t)


def pin_decode_constant_attention(orc):
    """q = 0 gives uniform attention 1/n_tau at step tau, so a token present since step 1 has
    A_j(t) = G * sum_{tau=1..t} gamma^(t - tau) / n_tau, and one appended at step u has the sum
    from tau = u; with n fixed this is the geometric series G/n (1 - gamma^k) / (1 - gamma)."""
    rng = np.random.default_rng(5)
    D, G, n0, gamma, steps = 8, 2, 7, 0.9, 12
    c = _random_cache(rng, n0, D, n0 + steps)
    for t in range(1, steps + 1):
        out = orc.decode_step(c, np.zeros((G, D)), rng.standard_normal(D), rng.standard_normal(D),
                              100 + t, gamma, 0.25)
        # uniform weights: every head outputs the plain mean of V
        np.testing.assert_allclose(out, np.tile(c.V[:c.n].mean(0), (G, 1)), rtol=1e-12, atol=1e-13)
    for j in range(c.n):
        born = max(1, j - n0 + 1)  # stage-1 rows exist from step 1; row n0+u-1 is appended at step u
        expect = G * sum(gamma ** (steps - tau) / (n0 + tau) for tau in range(born, steps + 1))
        assert abs(c.score[j] - expect) <= 1e-12 * expect, j


def pin_decode_special_cases(orc):
    """An empty cache returns v_new with score G; a saturated query returns the matching row;
    appending past the capacity is refused."""
    rng = np.random.default_rng(6)
    D, G = 16, 4
    c = O.UnitCache(3, D)
    vn = rng.standard_normal(D)
    out = orc.decode_step(c, rng.standard_normal((G, D)), rng.standard_normal(D), vn, 0, 0.9, 0.25)
    np.testing.assert_allclose(out, np.tile(vn, (G, 1)), rtol=1e-15)
    assert c.n == 1 and abs(c.score[0] - G) < 1e-15
    c = _random_cache(rng, 6, D, 7)
    kdir = c.K[2] / np.linalg.norm(c.K[2])
    q = np.tile(kdir * 400.0, (G, 1))
    out = orc.decode_step(c, q, np.zeros(D), np.zeros(D), 9, 0.9, 1.0)
    np.testing.assert_allclose(out, np.tile(c.V[2], (G, 1)), rtol=1e-6, atol=1e-6)
    try:
        orc.decode_step(c, q, np.zeros(D), np.zeros(D), 10, 0.9, 1.0)
    except O.OracleError as e:
        assert e.code == O.ECAPACITY
    else:
        raise AssertionError("append past capacity accepted")


# ----------------------------------------------------------------------------- evict

def pin_evict_hand(orc):
    """Hand-worked evictions: tie to the lower position, N = 0 (StreamingLLM) and a no-op."""
    g = _golden("evict_hand.json")
    D = 3
    for case in g["cases"]:
        n = g["n"]
        K = np.arange(n * D, dtype=float).reshape(n, D)
        c = O.UnitCache.from_rows(n, K, -K, g["pos"], g["score"])
        margin, kept = orc.evict(c, case["budget"])
        assert c.n == len(case["expected_pos"])
        np.testing.assert_array_equal(c.pos[:c.n], case["expected_pos"])
        np.testing.assert_array_equal(c.score[:c.n], case["expected_score"])
        assert margin == _num(case["expected_margin"]), (case, margin)
        src = np.array(case["expected_pos"]) - 100
        np.testing.assert_array_equal(c.K[:c.n], K[src])
        np.testing.assert_array_equal(c.V[:c.n], -K[src])


def _brute_force_keep(score, pos, T, M, N):
    """All N-subsets of the middle: the maximal score sum, then the lexicographically smallest
    sorted positions."""
    n = len(score)
    mid = list(range(T, n - M))
    best = None
    for sub in itertools.combinations(mid, N):
        key = (-sum(score[j] for j in sub), sorted(pos[j] for j in sub))
        if best is None or key < best[0]:
            best = (key, sub)
    return sorted(list(range(T)) + list(best[1]) + list(range(n - M, n)))


def pin_evict_bruteforce(orc):
    """Tiny inputs: the kept set equals brute-force search over all N-subsets (scores drawn from a
    few dyadic values, so sums are exact and ties are frequent)."""
    rng = np.random.default_rng(7)
    for trial in range(40):
        n = int(rng.integers(6, 17))
        budget = int(rng.integers(5, n))
        M = math.floor(float(np.float32(0.2)) * budget)
        N = budget - 4 - M
        if N < 0:
            continue
        score = rng.integers(0, 4, n) / 4.0
        pos = np.sort(rng.choice(1000, n, replace=False)).astype(np.int32)
        c = O.UnitCache.from_rows(n, np.arange(n, dtype=float)[:, None], np.zeros((n, 1)), pos, score)
        orc.evict(c, budget)
        expect = _brute_force_keep(score, pos, 4, M, N)
        np.testing.assert_array_equal(c.pos[:c.n], pos[expect])
        np.testing.assert_array_equal(c.K[:c.n, 0], np.array(expect, float))


def pin_evict_invariants(orc):
    """Random units: the cache ends at exactly the budget, sinks and the recent window survive,
    order is kept, rows move with their K, V, score and position, and every evicted history row
    scores no higher than every kept one."""
    rng = np.random.default_rng(8)
    for trial in range(30):
        D = 4
        n = int(rng.integers(10, 300))
        budget = int(rng.integers(5, n + 20))
        recent_frac = float(rng.choice([0.2, 0.1, 0.5]))
        M = math.floor(float(np.float32(recent_frac)) * budget)
        if budget - 4 - M < 0:
            continue
        K = rng.standard_normal((n, D))
        V = rng.standard_normal((n, D))
        score = rng.random(n)
        pos = np.arange(n, dtype=np.int32) * 3 + 11
        c = O.UnitCache.from_rows(n + 5, K, V, pos, score)
        margin, kept = orc.evict(c, budget, recent_frac=recent_frac)
        m = min(n, budget)
        assert c.n == m
        idx = (c.pos[:m] - 11) // 3
        assert np.all(np.diff(idx) > 0)
        np.testing.assert_array_equal(c.K[:m], K[idx])
        np.testing.assert_array_equal(c.V[:m], V[idx])
        np.testing.assert_array_equal(c.score[:m], score[idx])
        if n > budget:
            assert set(range(4)) <= set(idx) and set(range(n - M, n)) <= set(idx)
            hist_kept = [j for j in idx if 4 <= j < n - M]
            hist_drop = [j for j in range(4, n - M) if j not in set(idx)]
            assert len(hist_kept) == budget - 4 - M
            if hist_kept and hist_drop:
                assert min(score[hist_kept]) >= max(score[hist_drop])
                assert margin == min(score[hist_kept]) - max(score[hist_drop])
        else:
            assert np.array_equal(idx, np.arange(n)) and kept.all()
    try:
        orc.evict(O.UnitCache.from_rows(12, np.zeros((12, 2)), np.zeros((12, 2)), np.arange(12)), 3)
    except O.OracleError as e:
        assert e.code == O.EINVAL
    else:
        raise AssertionError("budget below T + M accepted")


def pin_evict_fill_hand(orc):
    """Hand-worked hole-filling eviction on a cache out of time order, the ordered eviction of the
    same slots, and the StreamingLLM policy with hole filling."""
    g = _golden("evict_fill_hand.json")
    n, D = g["n"], 2
    K = np.array([[j, 10.0 * j] for j in range(n)])
    for key, kw in (("fill", dict(fill=True)), ("ordered", dict(fill=False)),
                    ("streaming_fill", dict(fill=True, history=False))):
        case = g[key]
        c = O.UnitCache.from_rows(n, K, -K, g["pos"], g["score"])
        margin, kept = orc.evict(c, g["budget"], sink=g["sink"], recent_frac=g["recent_frac"], **kw)
        src = case["expected_src"]
        assert c.n == g["budget"]
        np.testing.assert_array_equal(c.pos[:c.n], case["expected_pos"])
        np.testing.assert_array_equal(c.score[:c.n], np.array(g["score"])[src])
        np.testing.assert_array_equal(c.K[:c.n], K[src])
        np.testing.assert_array_equal(c.V[:c.n], -K[src])
        assert margin == _num(case["expected_margin"]), (key, margin)
        if "expected_kept" in case:
            np.testing.assert_array_equal(kept.astype(int), case["expected_kept"])
            np.testing.assert_array_equal(c.score[:c.n], case["expected_score"])


def pin_evict_fill_matches_ordered_in_time_order(orc):
    """On a cache in time order, hole filling keeps exactly the rows the ordered compaction keeps
    (with and without history). It leaves every kept row below the budget in place, moves at most
    n - budget rows, and each row moves with its K, V, score and position."""
    rng = np.random.default_rng(11)
    for trial in range(40):
        D = 3
        n = int(rng.integers(8, 200))
        budget = int(rng.integers(5, n + 10))
        frac = float(rng.choice([0.2, 0.1, 0.5]))
        history = bool(rng.integers(0, 2))
        M = math.floor(float(np.float32(frac)) * budget) if history else budget - 4
        if budget - 4 - M < 0:
            continue
        K = rng.standard_normal((n, D))
        score = rng.integers(0, 8, n) / 8.0
        pos = np.sort(rng.choice(10 * n, n, replace=False)).astype(np.int32)
        a = O.UnitCache.from_rows(n, K, 2 * K, pos, score)
        b = O.UnitCache.from_rows(n, K, 2 * K, pos, score)
        ma, ka = orc.evict(a, budget, recent_frac=frac, history=history)
        mb, kb = orc.evict(b, budget, recent_frac=frac, history=history, fill=True)
        assert a.n == b.n == min(n, budget) and ma == mb
        np.testing.assert_array_equal(ka, kb)
        np.testing.assert_array_equal(np.sort(b.pos[:b.n]), a.pos[:a.n])
        src = np.searchsorted(pos, b.pos[:b.n])
        np.testing.assert_array_equal(b.K[:b.n], K[src])
        np.testing.assert_array_equal(b.V[:b.n], 2 * K[src])
        np.testing.assert_array_equal(b.score[:b.n], score[src])
        stay = kb[:b.n]
        np.testing.assert_array_equal(src[stay], np.nonzero(stay)[0])
        assert int((src != np.arange(b.n)).sum()) <= max(0, n - budget)


def pin_evict_fill_bruteforce_scrambled(orc):
    """Tiny caches whose slots are a random permutation of time order: hole filling keeps the set
    brute-force search keeps on the time-ordered cache (sinks and recents by position, the best
    N-subset of the rest with ties to lower positions)."""
    rng = np.random.default_rng(12)
    for trial in range(40):
        n = int(rng.integers(6, 14))
        budget = int(rng.integers(5, n))
        M = math.floor(float(np.float32(0.2)) * budget)
        N = budget - 4 - M
        if N < 0:
            continue
        score = rng.integers(0, 4, n) / 4.0
        pos = np.sort(rng.choice(1000, n, replace=False)).astype(np.int32)
        expect = set(pos[_brute_force_keep(score, pos, 4, M, N)])
        perm = rng.permutation(n)
        c = O.UnitCache.from_rows(n, perm[:, None].astype(float), np.zeros((n, 1)), pos[perm], score[perm])
        orc.evict(c, budget, fill=True)
        assert set(c.pos[:c.n]) == expect
        np.testing.assert_array_equal(pos[c.K[:c.n, 0].astype(int)], c.pos[:c.n])


def pin_evict_streaming(orc):
    """Without history the kept rows are the T lowest and the budget - T highest positions, in
    either compaction (the StreamingLLM baseline)."""
    rng = np.random.default_rng(13)
    for trial in range(30):
        n = int(rng.integers(6, 100))
        budget = int(rng.integers(4, n + 5))
        pos = rng.choice(5 * n, n, replace=False).astype(np.int32)
        score = rng.random(n)
        order = np.sort(pos)
        expect = set(order[:4]) | set(order[n - (budget - 4):]) if n > budget else set(pos)
        c = O.UnitCache.from_rows(n, np.zeros((n, 1)), np.zeros((n, 1)), pos, score)
        margin, _ = orc.evict(c, budget, history=False, fill=True)
        assert set(c.pos[:c.n]) == expect and margin == math.inf
        srt = np.argsort(pos)
        c = O.UnitCache.from_rows(n, np.zeros((n, 1)), np.zeros((n, 1)), pos[srt], score[srt])
        orc.evict(c, budget, history=False)
        assert set(c.pos[:c.n]) == expect


# ----------------------------------------------------------------------------- whole unit

def pin_run_unit_identity(orc):
    """Whole path with length-1 spans (stage 1 = identity), gamma = 1 and no eviction: every step
    is full attention over the prefill plus the appended tokens (torch SDPA)."""
    rng = np.random.default_rng(9)
    D, G, in_len, steps = 16, 2, 30, 8
    xk = _bf16(rng.standard_normal((in_len, D)))
    xv = _bf16(rng.standard_normal((in_len, D)))
    ss = list(range(3, 25))
    q = rng.standard_normal((steps, G, D))
    kn = rng.standard_normal((steps, D))
    vn = rng.standard_normal((steps, D))
    r = orc.run_unit(xk, xv, in_len, 3, 22, ss, [s + 1 for s in ss], [1] * len(ss), q=q, k_new=kn,
                     v_new=vn, new_pos=in_len + np.arange(steps), gamma=1.0, scale=D ** -0.5,
                     interval=steps + 1, budget=in_len, capacity=in_len + steps, cache_is_bf16=True)
    assert r["stage1_len"] == in_len and r["n"] == in_len + steps
    for t in range(steps):
        Kall = np.vstack([xk, kn[:t + 1]])
        Vall = np.vstack([xv, vn[:t + 1]])
        ref = torch.nn.functional.scaled_dot_product_attention(
            torch.from_numpy(q[t])[None, :, None, :],
            torch.from_numpy(Kall)[None, None].expand(1, G, -1, -1),
            torch.from_numpy(Vall)[None, None].expand(1, G, -1, -1))[0, :, 0].numpy()
        np.testing.assert_allclose(r["out"][t], ref, rtol=1e-10, atol=1e-12)
    np.testing.assert_array_equal(r["pos"], np.arange(in_len + steps))


def pin_run_unit_composition(orc):
    """run_unit equals stage1 + decode_step + evict called one by one, in the paper's order, under
    every eviction policy (with or without history, ordered or hole-filling compaction) and with
    other sink counts, recent fractions, decays and softmax scales."""
    for history, fill, sink, rf, gamma, scale in ((True, False, 4, 0.2, 0.9, 0.3), (False, False, 4, 0.2, 0.9, 0.3),
                                                  (True, True, 4, 0.2, 0.9, 0.3), (False, True, 4, 0.2, 0.9, 0.3),
                                                  (True, False, 2, 0.35, 0.97, 0.5), (True, True, 3, 0.3, 0.8, 0.2)):
        rng = np.random.default_rng(10)
        D, G, in_len, steps, interval, budget, cap = 8, 2, 50, 10, 4, 14, 60
        xk = _bf16(rng.standard_normal((in_len, D)))
        xv = _bf16(rng.standard_normal((in_len, D)))
        ss, se, sg = _random_spans(rng, 5, 40)
        q = rng.standard_normal((steps, G, D))
        kn, vn = _bf16(rng.standard_normal((steps, D))), _bf16(rng.standard_normal((steps, D)))
        npos = in_len + np.arange(steps)
        r = orc.run_unit(xk, xv, in_len, 5, 40, ss, se, sg, q=q, k_new=kn, v_new=vn, new_pos=npos,
                         gamma=gamma, scale=scale, interval=interval, budget=budget, capacity=cap,
                         cache_is_bf16=True, history=history, fill=fill, sink=sink, recent_frac=rf)
        sk = orc.stage1(xk, in_len, 5, 40, ss, se, sg, cache_is_bf16=True, capacity=cap)
        sv = orc.stage1(xv, in_len, 5, 40, ss, se, sg, cache_is_bf16=True, capacity=cap)
        c = O.UnitCache.from_rows(cap, sk["stored"], sv["stored"], sk["pos"])
        ev = 0
        for t in range(1, steps + 1):
            out = orc.decode_step(c, q[t - 1], kn[t - 1], vn[t - 1], npos[t - 1], gamma, scale)
            np.testing.assert_array_equal(out, r["out"][t - 1])
            if t % interval == 0:
                assert r["len_before"][ev] == c.n
                margin, _ = orc.evict(c, budget, sink, rf, history=history, fill=fill)
                assert margin == r["margin"][ev]
                np.testing.assert_array_equal(r["kept_pos"][ev][:c.n], c.pos[:c.n])
                ev += 1
        assert r["n"] == c.n
        np.testing.assert_array_equal(r["K"], c.K[:c.n])
        np.testing.assert_array_equal(r["pos"], c.pos[:c.n])
        np.testing.assert_array_equal(r["score"], c.score[:c.n])


ALL_PINS = [v for k, v in sorted(globals().items()) if k.startswith("pin_") and callable(v)]
