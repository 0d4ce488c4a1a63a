"""Eviction policies through voxzip_evict_ex against the oracle: hole-filling compaction on caches
out of time order, the StreamingLLM policy (no history), per-layer budgets, and gamma = 1; then
whole requests under each policy in lockstep with the oracle. Kept rows, positions, scores and K/V
bit-exact (the fill rule is deterministic on both sides)."""
import dataclasses
import math

import numpy as np
import pytest
import torch

import oracle
from gpu_harness import check_stage1, check_units, gpu_run, make_inputs, oracle_units, sample_units
from paper_2608_08569_gb300 import (DEV_BAD_POSITIONS, CacheDesc, allocate_cache, voxzip_evict_ex,
                                    voxzip_get_status)
from paper_2608_08569_gb300 import workloads as W

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def built():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2608_08569_gb300 import build
    build.build_library()
    oracle.build()
    voxzip_get_status()


def _scrambled_state(desc, lens, seed, ties):
    """Random rows and scores; each unit's positions are a random permutation of a sparse
    increasing sequence, so slot order is not time order."""
    g = torch.Generator(device="cuda")
    g.manual_seed(seed)
    c = allocate_cache(desc, "cuda")
    c["k"].copy_(torch.randn(c["k"].shape, generator=g, device="cuda").to(desc.dtype))
    c["v"].copy_(torch.randn(c["v"].shape, generator=g, device="cuda").to(desc.dtype))
    sc = torch.rand(c["score"].shape, generator=g, device="cuda") * 3
    c["score"].copy_(torch.floor(sc * 4) / 4 if ties else sc)
    base = torch.arange(desc.capacity, device="cuda", dtype=torch.int32) * 3 + 7
    perm = torch.argsort(torch.rand(c["pos"].shape, generator=g, device="cuda"), dim=-1)
    c["pos"].copy_(base[perm].to(torch.int32))
    c["len"].copy_(torch.as_tensor(lens, dtype=torch.int32, device="cuda").view(c["len"].shape))
    return c


def _unit(c, b, l, h, n, cap):
    f = lambda t: t.to("cpu", torch.float64).numpy()
    return oracle.UnitCache.from_rows(cap, f(c["k"][b, l, h, :n]), f(c["v"][b, l, h, :n]),
                                      c["pos"][b, l, h, :n].cpu().numpy(), f(c["score"][b, l, h, :n]))


def _compare(c, u, b, l, h):
    m = u.n
    assert int(c["len"][b, l, h]) == m, (b, l, h)
    np.testing.assert_array_equal(c["pos"][b, l, h, :m].cpu().numpy(), u.pos[:m], err_msg=str((b, l, h)))
    np.testing.assert_array_equal(c["score"][b, l, h, :m].double().cpu().numpy(), u.score[:m])
    np.testing.assert_array_equal(c["k"][b, l, h, :m].double().cpu().numpy(), u.K[:m])
    np.testing.assert_array_equal(c["v"][b, l, h, :m].double().cpu().numpy(), u.V[:m])


@pytest.mark.parametrize("dtype,D", [(torch.bfloat16, 128), (torch.float32, 64)])
@pytest.mark.parametrize("ties", [False, True])
@pytest.mark.parametrize("compaction", ["fill", "ordered"])
@pytest.mark.parametrize("per_layer", [False, True])
def test_evict_policies_random_states(dtype, D, ties, compaction, per_layer):
    B, L, H, C = 3, 2, 2, 2500
    desc = CacheDesc(B, L, 2 * H, H, D, C, dtype)
    rng = np.random.default_rng(30 + D + 2 * ties)
    budget = np.array([[7, 9], [300, 150], [2000, 1100]], np.int32)   # [B][L]; 2000: beyond one 1024 segment
    if not per_layer:
        budget[:, 1] = budget[:, 0]
    lens = np.stack([rng.integers(max(1, bb[0] - 20), min(C, 2 * bb[0] + 600), size=(L, H)) for bb in budget])
    lens[0, 0, 0] = budget[0, 0]                 # exactly at budget: untouched
    lens[2, 1, 1] = C                            # full cache
    lens[1, 0, 1] = budget[1, 0] + 1             # one row over
    c0 = _scrambled_state(desc, lens, seed=13 + D, ties=ties)
    if compaction == "ordered":                  # the ordered compaction assumes time order
        c0["pos"].copy_(torch.sort(c0["pos"], dim=-1).values)
    ref = {k: v.clone() for k, v in c0.items()}
    bud_t = torch.as_tensor(budget if per_layer else budget[:, 0].copy(), device="cuda")
    for sink, frac, history in ((4, 0.2, True), (0, 0.5, True), (2, 0.0, True), (4, 0.2, False), (1, 0.3, False)):
        c = {k: v.clone() for k, v in ref.items()}
        voxzip_evict_ex(desc, 0, L, c["k"], c["v"], c["score"], c["pos"], c["len"], bud_t, sink=sink,
                        recent_frac=frac, history=history, compaction=compaction)
        assert voxzip_get_status() == 0
        for b in range(B):
            for l in range(L):
                for h in range(H):
                    n = int(lens[b, l, h])
                    u = _unit(ref, b, l, h, n, C)
                    oracle.evict(u, int(budget[b, l]), sink=sink, recent_frac=frac, history=history,
                                 fill=compaction == "fill")
                    _compare(c, u, b, l, h)
                    if compaction == "fill" and n > budget[b, l]:
                        moved = (c["pos"][b, l, h, :u.n] != ref["pos"][b, l, h, :u.n]).sum().item()
                        assert moved <= n - budget[b, l]


def test_evict_fill_layer_range_and_duplicate_positions():
    """Only the requested layers are evicted; a unit whose positions repeat reports
    VOXZIP_DEV_BAD_POSITIONS instead of keeping a wrong count."""
    B, L, H, C, D = 1, 3, 1, 64, 64
    desc = CacheDesc(B, L, 2, H, D, C, torch.float32)
    lens = np.full((B, L, H), 40)
    c = _scrambled_state(desc, lens, seed=3, ties=False)
    ref = {k: v.clone() for k, v in c.items()}
    bud = torch.tensor([20], dtype=torch.int32, device="cuda")
    voxzip_evict_ex(desc, 1, 1, c["k"], c["v"], c["score"], c["pos"], c["len"], bud, compaction="fill")
    assert voxzip_get_status() == 0
    assert int(c["len"][0, 0, 0]) == 40 and int(c["len"][0, 2, 0]) == 40 and int(c["len"][0, 1, 0]) == 20
    assert torch.equal(c["pos"][0, 0], ref["pos"][0, 0]) and torch.equal(c["pos"][0, 2], ref["pos"][0, 2])
    c["pos"][0, 0, :40] = 5            # every position equal
    voxzip_evict_ex(desc, 0, 1, c["k"], c["v"], c["score"], c["pos"], c["len"], bud, compaction="fill")
    assert voxzip_get_status() & DEV_BAD_POSITIONS


def _pyramid(w):
    """Per-layer budgets falling linearly with depth around the workload's (PyramidKV-like)."""
    L = w.layers
    return [[max(w.sink + 4, int(round(bb * (1.5 - (l / max(1, L - 1)))))) for l in range(L)] for bb in w.budget]


POLICIES = {
    "fill": dict(compaction="fill"),
    "streaming": dict(history=False),
    "streaming_fill": dict(history=False, compaction="fill"),
    "per_layer": None,     # filled per workload
    "per_layer_fill": None,
}


@pytest.mark.parametrize("name,k", [("tiny_identity", 4), ("short", 16)])
@pytest.mark.parametrize("policy", list(POLICIES) + ["gamma1"])
def test_whole_path_under_policy(name, k, policy):
    w = W.CONFIGS[name]
    pol = POLICIES.get(policy)
    if policy.startswith("per_layer"):
        pol = dict(budget_bl=_pyramid(w), compaction="fill" if policy.endswith("fill") else "ordered")
    if policy == "gamma1":      # H2O-style accumulation: no decay
        w = dataclasses.replace(w, gamma=1.0)
        pol = None
    inp = make_inputs(w, "cuda")
    sample = sample_units(w, k)
    rec = gpu_run(w, inp, sample, policy=pol)
    check_stage1(w, inp, rec, sample)
    orc = oracle_units(w, inp, sample, policy=pol)
    diverged = check_units(w, rec, orc, sample, policy=pol)
    assert len(diverged) <= max(1, len(sample) // 8), diverged
