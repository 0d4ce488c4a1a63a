"""The C-ABI library builds for sm_103a, loads, exports every symbol include/voxzip.h declares,
and rejects invalid arguments synchronously (before any CUDA call, so these run without a GPU)."""
import ctypes
import os
import re

import pytest
import torch

from paper_2608_08569_gb300 import build as B

HEADER = os.path.join(B.ROOT, "include", "voxzip.h")


@pytest.fixture(scope="module")
def L():
    B.build_library()
    import paper_2608_08569_gb300 as V
    return V.lib()


def declared_functions():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(voxzip_[a-z_0-9]+)\s*\(", text)))


def test_header_declares_the_three_entry_points():
    names = declared_functions()
    for n in ("voxzip_anchor_fuse", "voxzip_decode_step", "voxzip_evict"):
        assert n in names


def test_library_exports_every_declared_symbol(L):
    missing = [n for n in declared_functions() if not hasattr(L, n)]
    assert not missing, missing


def test_checked_variant_builds_and_exports_every_declared_symbol():
    """The range-checked build (-DVOXZIP_CHECKED) compiles its guarded accesses, which the regular
    build leaves out, and exports the same C ABI."""
    path = B.build_library(checked=True)
    assert path == B.CHECKED_LIB_PATH and path != B.LIB_PATH
    lib = ctypes.CDLL(path)
    missing = [n for n in declared_functions() if not hasattr(lib, n)]
    assert not missing, missing


def test_library_is_sm103a_shared_object(L):
    assert os.path.dirname(B.LIB_PATH) == os.path.dirname(os.path.abspath(B.__file__))
    assert L.voxzip_version() == 100


def _desc(**kw):
    import paper_2608_08569_gb300 as V
    base = dict(batch=1, layers=2, q_heads=8, kv_heads=2, head_dim=128, capacity=64, dtype=1)
    base.update(kw)
    return V._native._Desc(*[base[k] for k in ("batch", "layers", "q_heads", "kv_heads", "head_dim",
                                                   "capacity", "dtype")])


P = ctypes.c_void_p(256)  # a non-null, 256-byte aligned stand-in; never dereferenced on these paths


@pytest.mark.parametrize("kw", [dict(head_dim=96), dict(q_heads=6, kv_heads=4), dict(batch=0), dict(dtype=7),
                                dict(capacity=0), dict(layers=-1)])
def test_bad_descriptor_is_einval(L, kw):
    d = _desc(**kw)
    rc = L.voxzip_decode_step(ctypes.byref(d), 0, 1, P, P, P, P, P, P, P, P, P, 0.9, 0.0, 0, P, None)
    assert rc == 1
    rc = L.voxzip_evict(ctypes.byref(d), 0, 1, P, P, P, P, P, P, 4, 0.2, None)
    assert rc == 1
    assert L.voxzip_anchor_fuse_workspace_size(ctypes.byref(d), 100, 4) == 0


def test_decode_argument_checks(L):
    d = _desc()
    ok = (P,) * 9
    assert L.voxzip_decode_step(None, 0, 1, *ok, 0.9, 0.0, 0, P, None) == 1
    assert L.voxzip_decode_step(ctypes.byref(d), 1, 2, *ok, 0.9, 0.0, 0, P, None) == 1   # layers out of range
    assert L.voxzip_decode_step(ctypes.byref(d), 0, 0, *ok, 0.9, 0.0, 0, P, None) == 1   # empty range
    for g in (0.0, -0.5, 1.5, float("nan")):
        assert L.voxzip_decode_step(ctypes.byref(d), 0, 1, *ok, g, 0.0, 0, P, None) == 1
    assert L.voxzip_decode_step(ctypes.byref(d), 0, 1, None, *ok[1:], 0.9, 0.0, 0, P, None) == 1
    assert L.voxzip_decode_step(ctypes.byref(d), 0, 1, ctypes.c_void_p(258), *ok[1:], 0.9, 0.0, 0, P,
                                None) == 1  # misaligned q
    assert L.voxzip_decode_step(ctypes.byref(d), 0, 1, *ok, 0.9, float("inf"), 0, P, None) == 1
    d17 = _desc(q_heads=34, kv_heads=2)  # group of 17 > 16
    assert L.voxzip_decode_step(ctypes.byref(d17), 0, 1, *ok, 0.9, 0.0, 0, P, None) == 2


def test_evict_argument_checks(L):
    d = _desc()
    assert L.voxzip_evict(ctypes.byref(d), 0, 1, P, P, P, P, P, P, -1, 0.2, None) == 1     # sink < 0
    assert L.voxzip_evict(ctypes.byref(d), 0, 1, P, P, P, P, P, P, 4, 1.5, None) == 1      # recent_frac > 1
    assert L.voxzip_evict(ctypes.byref(d), 0, 1, P, P, P, P, P, None, 4, 0.2, None) == 1   # no budget
    assert L.voxzip_evict(ctypes.byref(d), 2, 1, P, P, P, P, P, P, 4, 0.2, None) == 1      # layer range


def test_anchor_fuse_argument_checks(L):
    d = _desc()
    need = L.voxzip_anchor_fuse_workspace_size(ctypes.byref(d), 100, 10)
    assert need > 0 and need % 256 == 0
    args = lambda **o: [o.get(k, v) for k, v in [
        ("kp", P), ("vp", P), ("stride", 100), ("in_len", P), ("ab", P), ("al", P), ("off", P), ("ns", 10),
        ("ss", P), ("se", P), ("sg", P), ("ak", None), ("av", None), ("astr", 0), ("kc", P), ("vc", P), ("sc", P),
        ("pos", P), ("len", P), ("sm", None), ("ws", P), ("wsb", need), ("stream", None)]]
    f = lambda **o: L.voxzip_anchor_fuse(ctypes.byref(d), *args(**o))
    assert f(wsb=need - 1) == 1                  # workspace too small
    assert f(ws=ctypes.c_void_p(16)) == 1        # workspace not 256-byte aligned
    assert f(ak=P) == 1                          # one anchor pointer without the other
    assert f(ak=P, av=P, astr=0) == 1            # anchors without a stride
    assert f(stride=0) == 1
    assert f(ns=-1) == 1
    assert f(ss=None) == 1                       # spans missing while num_spans > 0
    assert f(kp=None) == 1


def test_status_strings(L):
    for code, name in enumerate(["VOXZIP_OK", "VOXZIP_EINVAL", "VOXZIP_EUNSUPPORTED", "VOXZIP_ECUDA"]):
        assert L.voxzip_status_string(code).decode() == name


def test_binding_rejects_host_tensors():
    import paper_2608_08569_gb300 as V
    desc = V.CacheDesc(1, 1, 2, 1, 64, 8, torch.float32)
    t = torch.zeros(1, 1, 1, 8, 64)
    with pytest.raises(ValueError):
        V.voxzip_evict(desc, 0, 1, t, t, torch.zeros(1, 1, 1, 8), torch.zeros(1, 1, 1, 8, dtype=torch.int32),
                       torch.zeros(1, 1, 1, dtype=torch.int32), torch.zeros(1, dtype=torch.int32))


# --------------------------------------------------------------------- the NEXT rows' entry points

def _paged(**kw):
    import paper_2608_08569_gb300 as V
    base = dict(k_pool=256, v_pool=256, page_table=256, free_pages=256, free_count=256, pages=64, max_pages=1)
    base.update(kw)
    return V._native._Paged(*[base[k] for k in ("k_pool", "v_pool", "page_table", "free_pages", "free_count",
                                                   "pages", "max_pages")])


def _policy(**kw):
    import paper_2608_08569_gb300 as V
    base = dict(sink=4, recent_frac=0.2, history=1, budget_stride_b=1, budget_stride_l=0, compaction=0)
    base.update(kw)
    return V._native._EvictPolicy(*[base[k] for k in ("sink", "recent_frac", "history", "budget_stride_b",
                                                         "budget_stride_l", "compaction")])


@pytest.mark.parametrize("kw", [dict(compaction=2), dict(history=3), dict(budget_stride_b=-1), dict(sink=-1),
                                dict(recent_frac=1.5)])
def test_evict_policy_is_validated(L, kw):
    d, pol = _desc(), _policy(**kw)
    assert L.voxzip_evict_ex(ctypes.byref(d), 0, 1, P, P, P, P, P, P, ctypes.byref(pol), None) == 1
    assert L.voxzip_evict_ex(ctypes.byref(d), 0, 1, P, P, P, P, P, P, None, None) == 1


@pytest.mark.parametrize("kw", [dict(max_pages=2), dict(pages=1), dict(k_pool=0), dict(k_pool=264)])
def test_paged_cache_is_validated(L, kw):
    """capacity (64 here) must be 64 x max_pages, the pool must hold a page per unit, pools are
    non-null and 16-byte aligned."""
    d, pc = _desc(), _paged(**kw)
    assert L.voxzip_decode_step_paged(ctypes.byref(d), ctypes.byref(pc), 0, 1, P, P, P, P, P, P, P, 0.9, 0.0, 0,
                                      P, None) == 1
    assert L.voxzip_paged_init(ctypes.byref(d), ctypes.byref(pc), P, None) == 1
    pol = _policy()
    assert L.voxzip_evict_paged(ctypes.byref(d), ctypes.byref(pc), 0, 1, P, P, P, P, ctypes.byref(pol), None) == 1


def test_paged_init_needs_lengths(L):
    d, pc = _desc(), _paged()
    assert L.voxzip_paged_init(ctypes.byref(d), ctypes.byref(pc), None, None) == 1


@pytest.mark.parametrize("d_model,dtype,keep", [(12, 1, 1), (6, 0, 1), (64, 1, 2), (0, 1, 1)])
def test_embed_fuse_is_validated(L, d_model, dtype, keep):
    import paper_2608_08569_gb300 as V
    e = V._native._EmbedDesc(2, d_model, 64, dtype)
    assert L.voxzip_embed_fuse_workspace_size(ctypes.byref(e), 100, 3) == 0 or keep == 2
    rc = L.voxzip_embed_fuse(ctypes.byref(e), P, 100, P, P, P, P, 0, None, None, None, None, 0, keep, P, P, P,
                             None, P, 1 << 20, None)
    assert rc == 1


@pytest.mark.parametrize("limit", [0, (1 << 20) + 1])
def test_selftest_limit_is_validated(L, limit):
    assert L.voxzip_selftest_bounded_wait(limit, None) == 1


@pytest.mark.parametrize("ptr,nbytes,sink", [(0, 256, 256), (264, 256, 256), (256, 100, 256), (256, 256, 0)])
def test_stream_read_is_validated(L, ptr, nbytes, sink):
    """The streaming-read measurement helper rejects a null or unaligned buffer, a size that is not
    a multiple of 16 and a null sink before touching the device."""
    assert L.voxzip_stream_read(ctypes.c_void_p(ptr) if ptr else None, nbytes,
                                ctypes.c_void_p(sink) if sink else None, None) == 1


def test_prefill_may_be_pinned_host_memory_other_tensors_not():
    """The binding accepts the prefilled K/V in pinned host memory (stage 1 then streams them over
    the host link) and still demands device tensors for every other argument."""
    import torch
    from paper_2608_08569_gb300 import _native as N
    if not torch.cuda.is_available():
        # without a CUDA runtime no host memory can be pinned; the check on a plain CPU tensor stands
        with pytest.raises(ValueError, match="pinned host memory"):
            N._need(torch.zeros(4, dtype=torch.bfloat16), "k_prefill", torch.bfloat16, pinned_ok=True)
    with pytest.raises(ValueError, match="on a CUDA device"):
        N._need(torch.zeros(4, dtype=torch.int32), "in_len", torch.int32)
