"""voxzip_anchor_fuse_noalloc, the stage-1 entry point for callers that cannot allocate device
memory (for example a runtime whose device memory all belongs to another framework's pool, or an
audio front-end that must not allocate while serving), against the regular voxzip_anchor_fuse.

Both are called through the C ABI on the same seeded inputs; the cache they produce must agree
exactly (stage-1 rows are bit-exact between the library and the oracle, so the tolerance is
zero). Two calls of the allocation-free entry point run back to back on different workloads, so a
stale scratch from the first call would show in the second. Needs a GB300.
"""
import ctypes

import numpy as np
import pytest
import torch

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def built():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2608_08569_gb300 import build
    build.build_library()


def _inputs(w, anchors):
    from gpu_harness import make_anchors
    from paper_2608_08569_gb300 import workloads as W
    sp = W.make_spans(w)
    k, v = W.make_prefill(w, "cuda")
    i32 = lambda a: torch.as_tensor(np.asarray(a), dtype=torch.int32, device="cuda")
    args = (k, v, i32(w.in_len), i32([w.audio_begin] * w.batch), i32(w.audio_len), i32(sp.off), i32(sp.start),
            i32(sp.end), i32(sp.groups))
    anc = make_anchors(w, sp, "cuda") if anchors else (None, None)
    return args, anc


def _fuse(w, args, anc, noalloc):
    import paper_2608_08569_gb300 as V
    desc = V.CacheDesc(w.batch, w.layers, w.q_heads, w.kv_heads, w.head_dim, w.capacity, w.dtype)
    c = V.allocate_cache(desc)
    c["len"].fill_(-7)     # both entry points must overwrite every length
    c["pos"].fill_(-7)
    sm = torch.full((w.batch, w.stride), -7, dtype=torch.int32, device="cuda")
    fn = V.voxzip_anchor_fuse_noalloc if noalloc else V.voxzip_anchor_fuse
    fn(desc, *args, c["k"], c["v"], c["score"], c["pos"], c["len"], slot_map=sm, anchor_k=anc[0], anchor_v=anc[1])
    torch.cuda.synchronize()
    assert V.voxzip_get_status() == 0
    c["slot_map"] = sm
    return c


def test_noalloc_matches_the_workspace_entry_point_on_two_calls_in_a_row():
    from paper_2608_08569_gb300 import workloads as W
    cases = [(W.scaled(W.CONFIGS["batched"], layers=2, batch=8, name="batched_small"), False),
             (W.scaled(W.CONFIGS["stress"], layers=1, batch=2, name="stress_small"), True),
             (W.CONFIGS["tiny"], False)]
    for w, anchors in cases:
        args, anc = _inputs(w, anchors)
        ref = _fuse(w, args, anc, noalloc=False)
        got = _fuse(w, args, anc, noalloc=True)
        n = int(ref["len"].max())
        assert n > 0 and torch.equal(ref["len"], got["len"]), w.name
        assert torch.equal(ref["slot_map"], got["slot_map"]), w.name
        for key in ("k", "v", "score", "pos"):
            assert torch.equal(ref[key][..., :n], got[key][..., :n]) if key in ("score", "pos") else \
                torch.equal(ref[key][:, :, :, :n], got[key][:, :, :, :n]), (w.name, key)


def test_noalloc_rejects_requests_larger_than_its_scratch():
    import paper_2608_08569_gb300 as V
    L = V.lib()
    d = V._native._Desc(64, 1, 2, 1, 64, 8, 1)
    assert L.voxzip_anchor_fuse_workspace_size(ctypes.byref(d), 20000, 0) > (4 << 20)
    p = ctypes.c_void_p(256)
    rc = L.voxzip_anchor_fuse_noalloc(ctypes.byref(d), p, p, 20000, p, p, p, p, 0, None, None, None, None, None, 0,
                                      p, p, p, p, p, None, None)
    assert rc == V.VOXZIP_ESCRATCH


def _limit_case(stride):
    """One sequence of `stride` audio tokens in spans of four (one group each), 64-wide fp32 rows."""
    import paper_2608_08569_gb300 as V
    n_spans = stride // 4
    desc = V.CacheDesc(1, 1, 1, 1, 64, n_spans + 8, torch.float32)
    g = torch.Generator(device="cuda")
    g.manual_seed(5)
    k = torch.randn(1, 1, 1, stride, 64, generator=g, device="cuda")
    v = torch.randn(1, 1, 1, stride, 64, generator=g, device="cuda")
    i32 = lambda a: torch.as_tensor(np.asarray(a), dtype=torch.int32, device="cuda")
    starts = np.arange(n_spans) * 4
    args = (k, v, i32([stride]), i32([0]), i32([stride]), i32([0, n_spans]), i32(starts), i32(starts + 4),
            i32(np.ones(n_spans)))
    return desc, args


def _largest_stride_within(limit):
    """The largest prefill stride (multiple of 4, one span per four tokens) whose workspace fits."""
    import paper_2608_08569_gb300 as V
    desc = V.CacheDesc(1, 1, 1, 1, 64, 8, torch.float32)
    lo, hi = 4, 1 << 22
    while hi - lo > 4:
        mid = (lo + hi) // 8 * 4
        if V.voxzip_anchor_fuse_workspace_size(desc, mid, mid // 4) <= limit:
            lo = mid
        else:
            hi = mid
    return lo


def test_noalloc_accepts_a_request_just_under_its_scratch_and_rejects_one_just_over():
    import paper_2608_08569_gb300 as V
    limit = 4 << 20
    stride = _largest_stride_within(limit)
    desc, args = _limit_case(stride)
    assert limit - 4096 < V.voxzip_anchor_fuse_workspace_size(desc, stride, stride // 4) <= limit
    outs = []
    for noalloc in (False, True):
        c = V.allocate_cache(desc)
        c["len"].fill_(-7)
        sm = torch.full((1, stride), -7, dtype=torch.int32, device="cuda")
        fn = V.voxzip_anchor_fuse_noalloc if noalloc else V.voxzip_anchor_fuse
        fn(desc, *args, c["k"], c["v"], c["score"], c["pos"], c["len"], slot_map=sm)
        torch.cuda.synchronize()
        assert V.voxzip_get_status() == 0
        c["slot_map"] = sm
        outs.append(c)
    ref, got = outs
    n = stride // 4
    assert int(ref["len"][0, 0, 0]) == n and torch.equal(ref["len"], got["len"])
    assert torch.equal(ref["slot_map"], got["slot_map"])
    for key in ("k", "v"):
        assert torch.equal(ref[key][:, :, :, :n], got[key][:, :, :, :n]), key
    for key in ("score", "pos"):
        assert torch.equal(ref[key][..., :n], got[key][..., :n]), key
    # four more tokens (and one more span) take the request past the fixed scratch
    desc2, args2 = _limit_case(stride + 4)
    assert V.voxzip_anchor_fuse_workspace_size(desc2, stride + 4, (stride + 4) // 4) > limit
    c = V.allocate_cache(desc2)
    with pytest.raises(V.VoxZipError) as e:
        V.voxzip_anchor_fuse_noalloc(desc2, *args2, c["k"], c["v"], c["score"], c["pos"], c["len"])
    assert e.value.code == V.VOXZIP_ESCRATCH
