"""ctypes binding of ``libvoxzip.so`` (declared in ``include/voxzip.h``).

Argument marshalling only: tensors become device pointers, the current torch stream becomes the
launch stream, and a non-OK status becomes an exception. Every step of the path runs in the
library's CUDA kernels; there is no fallback when the library is missing.
"""
from __future__ import annotations

import ctypes
import os
import threading
from dataclasses import dataclass

import torch

from .build import CHECKED_LIB_PATH
from .build import LIB_PATH as _REGULAR_LIB_PATH

# VOXZIP_CHECKED=1 selects the range-checked build (kernels report out-of-range accesses as
# DEV_BOUNDS instead of making them); it is slower and meant for tests.
LIB_PATH = CHECKED_LIB_PATH if os.environ.get("VOXZIP_CHECKED", "0") not in ("", "0") else _REGULAR_LIB_PATH

VOXZIP_OK, VOXZIP_EINVAL, VOXZIP_EUNSUPPORTED, VOXZIP_ECUDA, VOXZIP_ESCRATCH = 0, 1, 2, 3, 4
DEV_BAD_SPANS, DEV_CAPACITY, DEV_LEN_HINT, DEV_BAD_BUDGET, DEV_TIMEOUT = 0x1, 0x2, 0x4, 0x8, 0x10
DEV_BAD_POSITIONS, DEV_BOUNDS = 0x20, 0x40
VOXZIP_COMPACT_ORDERED, VOXZIP_COMPACT_FILL = 0, 1
VOXZIP_F32, VOXZIP_BF16 = 0, 1

_DTYPES = {torch.float32: VOXZIP_F32, torch.bfloat16: VOXZIP_BF16}


class VoxZipError(RuntimeError):
    def __init__(self, fn: str, code: int, text: str):
        super().__init__(f"{fn} failed: {text} ({code})")
        self.code = code


class _Desc(ctypes.Structure):
    _fields_ = [("batch", ctypes.c_int32), ("layers", ctypes.c_int32), ("q_heads", ctypes.c_int32),
                ("kv_heads", ctypes.c_int32), ("head_dim", ctypes.c_int32), ("capacity", ctypes.c_int32),
                ("dtype", ctypes.c_int32)]


@dataclass(frozen=True)
class CacheDesc:
    """Shape of a VoxZip cache: B sequences x L layers x Hkv kv-heads, C slots of D elements."""
    batch: int
    layers: int
    q_heads: int
    kv_heads: int
    head_dim: int
    capacity: int
    dtype: torch.dtype = torch.bfloat16

    @property
    def group(self) -> int:
        return self.q_heads // self.kv_heads

    def c_struct(self) -> _Desc:
        return _Desc(self.batch, self.layers, self.q_heads, self.kv_heads, self.head_dim, self.capacity,
                     _DTYPES[self.dtype])


class _EmbedDesc(ctypes.Structure):
    _fields_ = [("batch", ctypes.c_int32), ("d_model", ctypes.c_int32), ("capacity", ctypes.c_int32),
                ("dtype", ctypes.c_int32)]


@dataclass(frozen=True)
class EmbedDesc:
    """Shape of embedding-level stage 1: B sequences, output rows of d_model elements, C rows each."""
    batch: int
    d_model: int
    capacity: int
    dtype: torch.dtype = torch.bfloat16

    def c_struct(self) -> _EmbedDesc:
        return _EmbedDesc(self.batch, self.d_model, self.capacity, _DTYPES[self.dtype])


class _EvictPolicy(ctypes.Structure):
    _fields_ = [("sink", ctypes.c_int32), ("recent_frac", ctypes.c_float), ("history", ctypes.c_int32),
                ("budget_stride_b", ctypes.c_int32), ("budget_stride_l", ctypes.c_int32),
                ("compaction", ctypes.c_int32)]


class _Paged(ctypes.Structure):
    _fields_ = [("k_pool", ctypes.c_void_p), ("v_pool", ctypes.c_void_p), ("page_table", ctypes.c_void_p),
                ("free_pages", ctypes.c_void_p), ("free_count", ctypes.c_void_p), ("pages", ctypes.c_int32),
                ("max_pages", ctypes.c_int32)]


PAGE_TOKENS = 64

_lock = threading.Lock()
_lib = None
_vp = ctypes.c_void_p
_i32 = ctypes.c_int32
_f32 = ctypes.c_float
_sz = ctypes.c_size_t
_f64 = ctypes.c_double
_DP = ctypes.POINTER(_Desc)
_EP = ctypes.POINTER(_EmbedDesc)


def lib() -> ctypes.CDLL:
    """The loaded library; raises if it has not been built (no CPU fallback exists)."""
    global _lib
    with _lock:
        if _lib is None:
            if not os.path.exists(LIB_PATH):
                raise RuntimeError(f"{LIB_PATH} is missing: build it with paper_2608_08569_gb300.build")
            L = ctypes.CDLL(LIB_PATH)
            L.voxzip_anchor_fuse.argtypes = [_DP, _vp, _vp, _i32, _vp, _vp, _vp, _vp, _i32, _vp, _vp, _vp, _vp,
                                             _vp, _i32, _vp, _vp, _vp, _vp, _vp, _vp, _vp, _sz, _vp]
            L.voxzip_anchor_fuse_noalloc.argtypes = [_DP, _vp, _vp, _i32, _vp, _vp, _vp, _vp, _i32, _vp, _vp, _vp,
                                                     _vp, _vp, _i32, _vp, _vp, _vp, _vp, _vp, _vp, _vp]
            L.voxzip_anchor_fuse_noalloc.restype = _i32
            L.voxzip_anchor_fuse_workspace_size.argtypes = [_DP, _i32, _i32]
            L.voxzip_anchor_fuse_workspace_size.restype = _sz
            L.voxzip_decode_step.argtypes = [_DP, _i32, _i32, _vp, _vp, _vp, _vp, _vp, _vp, _vp, _vp, _vp,
                                             _f32, _f32, _i32, _vp, _vp]
            L.voxzip_evict.argtypes = [_DP, _i32, _i32, _vp, _vp, _vp, _vp, _vp, _vp, _i32, _f32, _vp]
            L.voxzip_get_status.argtypes = [ctypes.POINTER(ctypes.c_uint32), _vp]
            L.voxzip_evict_ex.argtypes = [_DP, _i32, _i32, _vp, _vp, _vp, _vp, _vp, _vp,
                                          ctypes.POINTER(_EvictPolicy), _vp]
            _PP = ctypes.POINTER(_Paged)
            L.voxzip_paged_init.argtypes = [_DP, _PP, _vp, _vp]
            L.voxzip_anchor_fuse_paged.argtypes = [_DP, _PP, _vp, _vp, _i32, _vp, _vp, _vp, _vp, _i32, _vp, _vp, _vp,
                                                   _vp, _vp, _i32, _vp, _vp, _vp, _vp, _vp, _sz, _vp]
            L.voxzip_anchor_fuse_paged_workspace_size.argtypes = [_DP, _i32, _i32]
            L.voxzip_anchor_fuse_paged_workspace_size.restype = _sz
            L.voxzip_decode_step_paged.argtypes = [_DP, _PP, _i32, _i32, _vp, _vp, _vp, _vp, _vp, _vp, _vp, _f32,
                                                   _f32, _i32, _vp, _vp]
            L.voxzip_evict_paged.argtypes = [_DP, _PP, _i32, _i32, _vp, _vp, _vp, _vp, ctypes.POINTER(_EvictPolicy),
                                             _vp]
            L.voxzip_selftest_bounded_wait.argtypes = [ctypes.c_uint32, _vp]
            L.voxzip_selftest_bounded_wait.restype = _i32
            L.voxzip_stream_read.argtypes = [_vp, _sz, _vp, _vp]
            L.voxzip_stream_read.restype = _i32
            L.voxzip_segments_to_spans.argtypes = [_i32, _vp, _vp, _vp, _vp, _f64, _i32, _i32, _f64, _vp, _vp, _vp,
                                                   _vp, _vp]
            L.voxzip_embed_fuse.argtypes = [_EP, _vp, _i32, _vp, _vp, _vp, _vp, _i32, _vp, _vp, _vp, _vp, _i32,
                                            _i32, _vp, _vp, _vp, _vp, _vp, _sz, _vp]
            L.voxzip_embed_fuse_workspace_size.argtypes = [_EP, _i32, _i32]
            L.voxzip_embed_fuse_workspace_size.restype = _sz
            L.voxzip_status_string.argtypes = [_i32]
            L.voxzip_status_string.restype = ctypes.c_char_p
            L.voxzip_version.restype = _i32
            for f in (L.voxzip_anchor_fuse, L.voxzip_decode_step, L.voxzip_evict, L.voxzip_get_status,
                      L.voxzip_segments_to_spans, L.voxzip_embed_fuse, L.voxzip_evict_ex, L.voxzip_paged_init,
                      L.voxzip_anchor_fuse_paged, L.voxzip_decode_step_paged, L.voxzip_evict_paged):
                f.restype = _i32
            _lib = L
    return _lib


def _check(fn: str, code: int) -> None:
    if code != VOXZIP_OK:
        raise VoxZipError(fn, code, lib().voxzip_status_string(code).decode())


def _ptr(t):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


def _stream(stream):
    s = torch.cuda.current_stream() if stream is None else stream
    return ctypes.c_void_p(s.cuda_stream)


def _need(t: torch.Tensor, name: str, dtype: torch.dtype, shape=None, pinned_ok: bool = False) -> None:
    """Checks a tensor argument; `pinned_ok` also accepts page-locked host memory (which the device
    addresses directly under unified addressing)."""
    if not isinstance(t, torch.Tensor):
        raise TypeError(f"{name} must be a torch.Tensor")
    if t.dtype != dtype:
        raise ValueError(f"{name}: dtype {t.dtype}, expected {dtype}")
    if not t.is_cuda and not (pinned_ok and t.is_pinned()):
        raise ValueError(f"{name} must be on a CUDA device" + (" or in pinned host memory" if pinned_ok else ""))
    if not t.is_contiguous():
        raise ValueError(f"{name} must be contiguous")
    if shape is not None and tuple(t.shape) != tuple(shape):
        raise ValueError(f"{name}: shape {tuple(t.shape)}, expected {tuple(shape)}")


def _check_cache(desc: CacheDesc, k_cache, v_cache, score, pos, len_) -> None:
    cs = (desc.batch, desc.layers, desc.kv_heads, desc.capacity)
    _need(k_cache, "k_cache", desc.dtype, cs + (desc.head_dim,))
    _need(v_cache, "v_cache", desc.dtype, cs + (desc.head_dim,))
    _need(score, "score", torch.float32, cs)
    _need(pos, "pos", torch.int32, cs)
    _need(len_, "len", torch.int32, cs[:3])


def allocate_cache(desc: CacheDesc, device="cuda"):
    """Device tensors for a cache of shape ``desc``: k, v, score, pos, len (zero-filled)."""
    cs = (desc.batch, desc.layers, desc.kv_heads, desc.capacity)
    return dict(k=torch.zeros(cs + (desc.head_dim,), dtype=desc.dtype, device=device),
                v=torch.zeros(cs + (desc.head_dim,), dtype=desc.dtype, device=device),
                score=torch.zeros(cs, dtype=torch.float32, device=device),
                pos=torch.zeros(cs, dtype=torch.int32, device=device),
                len=torch.zeros(cs[:3], dtype=torch.int32, device=device))


def allocate_paged_cache(desc: CacheDesc, pages: int, device="cuda", stream=None):
    """A paged cache: K and V page pools of `pages` pages of 64 rows, the page table and the free
    stack, and the dense per-slot state (score, pos, len). desc.capacity (a multiple of 64) bounds
    one unit. The cache starts empty (voxzip_paged_init)."""
    if desc.capacity % PAGE_TOKENS:
        raise ValueError("a paged cache's capacity must be a multiple of 64")
    cs = (desc.batch, desc.layers, desc.kv_heads, desc.capacity)
    mp = desc.capacity // PAGE_TOKENS
    pc = dict(k_pool=torch.zeros(pages, PAGE_TOKENS, desc.head_dim, dtype=desc.dtype, device=device),
              v_pool=torch.zeros(pages, PAGE_TOKENS, desc.head_dim, dtype=desc.dtype, device=device),
              page_table=torch.full(cs[:3] + (mp,), -1, dtype=torch.int32, device=device),
              free_pages=torch.zeros(pages, dtype=torch.int32, device=device),
              free_count=torch.zeros(1, dtype=torch.int32, device=device),
              score=torch.zeros(cs, dtype=torch.float32, device=device),
              pos=torch.zeros(cs, dtype=torch.int32, device=device),
              len=torch.zeros(cs[:3], dtype=torch.int32, device=device), pages=int(pages), max_pages=mp)
    voxzip_paged_init(desc, pc, stream=stream)
    return pc


def _paged_struct(desc: CacheDesc, pc) -> _Paged:
    mp = desc.capacity // PAGE_TOKENS
    _need(pc["k_pool"], "k_pool", desc.dtype, (pc["pages"], PAGE_TOKENS, desc.head_dim))
    _need(pc["v_pool"], "v_pool", desc.dtype, (pc["pages"], PAGE_TOKENS, desc.head_dim))
    _need(pc["page_table"], "page_table", torch.int32, (desc.batch, desc.layers, desc.kv_heads, mp))
    _need(pc["free_pages"], "free_pages", torch.int32, (pc["pages"],))
    _need(pc["free_count"], "free_count", torch.int32, (1,))
    return _Paged(pc["k_pool"].data_ptr(), pc["v_pool"].data_ptr(), pc["page_table"].data_ptr(),
                  pc["free_pages"].data_ptr(), pc["free_count"].data_ptr(), int(pc["pages"]), mp)


def _check_dense_state(desc: CacheDesc, score, pos, len_) -> None:
    cs = (desc.batch, desc.layers, desc.kv_heads, desc.capacity)
    _need(score, "score", torch.float32, cs)
    _need(pos, "pos", torch.int32, cs)
    _need(len_, "len", torch.int32, cs[:3])


def voxzip_paged_init(desc: CacheDesc, pc, stream=None) -> None:
    """Empties every unit of a paged cache (page u for unit u's slot 0, the rest free)."""
    d, ps = desc.c_struct(), _paged_struct(desc, pc)
    _need(pc["len"], "len", torch.int32, (desc.batch, desc.layers, desc.kv_heads))
    _check("voxzip_paged_init", lib().voxzip_paged_init(ctypes.byref(d), ctypes.byref(ps), _ptr(pc["len"]),
                                                        _stream(stream)))


def paged_pages_in_use(pc) -> int:
    """Pages held by units (synchronises with the device)."""
    return int(pc["pages"]) - int(pc["free_count"].item())


def voxzip_anchor_fuse_paged(desc: CacheDesc, pc, k_prefill, v_prefill, in_len, audio_begin, audio_len, span_off,
                             span_start, span_end, span_groups, *, slot_map=None, anchor_k=None, anchor_v=None,
                             workspace=None, stream=None) -> None:
    """Stage 1 (Sec. 3.2.1) into a paged cache: each unit returns its pages and takes the ones its
    stage-1 rows need."""
    B, L, H, D = desc.batch, desc.layers, desc.kv_heads, desc.head_dim
    stride = k_prefill.shape[3]
    _need(k_prefill, "k_prefill", desc.dtype, (B, L, H, stride, D), pinned_ok=True)
    _need(v_prefill, "v_prefill", desc.dtype, (B, L, H, stride, D), pinned_ok=True)
    for name, t in (("in_len", in_len), ("audio_begin", audio_begin), ("audio_len", audio_len)):
        _need(t, name, torch.int32, (B,))
    _need(span_off, "span_off", torch.int32, (B + 1,))
    num_spans = span_start.numel()
    for name, t in (("span_start", span_start), ("span_end", span_end), ("span_groups", span_groups)):
        _need(t, name, torch.int32, (num_spans,))
    _check_dense_state(desc, pc["score"], pc["pos"], pc["len"])
    if slot_map is not None:
        _need(slot_map, "slot_map", torch.int32, (B, stride))
    anchor_stride = 0
    if anchor_k is not None or anchor_v is not None:
        anchor_stride = anchor_k.shape[3]
        _need(anchor_k, "anchor_k", desc.dtype, (B, L, H, anchor_stride, D))
        _need(anchor_v, "anchor_v", desc.dtype, (B, L, H, anchor_stride, D))
    d, ps = desc.c_struct(), _paged_struct(desc, pc)
    need = int(lib().voxzip_anchor_fuse_paged_workspace_size(ctypes.byref(d), int(stride), int(num_spans)))
    if workspace is None or workspace.numel() < need:
        workspace = torch.empty(max(need, 256), dtype=torch.uint8, device=k_prefill.device)
    _need(workspace, "workspace", torch.uint8)
    _check("voxzip_anchor_fuse_paged", lib().voxzip_anchor_fuse_paged(
        ctypes.byref(d), ctypes.byref(ps), _ptr(k_prefill), _ptr(v_prefill), int(stride), _ptr(in_len),
        _ptr(audio_begin), _ptr(audio_len), _ptr(span_off), int(num_spans), _ptr(span_start), _ptr(span_end),
        _ptr(span_groups), _ptr(anchor_k), _ptr(anchor_v), int(anchor_stride), _ptr(pc["score"]), _ptr(pc["pos"]),
        _ptr(pc["len"]), _ptr(slot_map), _ptr(workspace), int(workspace.numel()), _stream(stream)))


def voxzip_decode_step_paged(desc: CacheDesc, pc, layer_begin: int, layer_count: int, q, k_new, v_new, new_pos,
                             gamma: float, out, *, sm_scale: float = 0.0, max_len: int = 0, stream=None) -> None:
    """One decode step (Eq. 1, Eq. 2, Eq. 6) on a paged cache."""
    B, Hq, H, D = desc.batch, desc.q_heads, desc.kv_heads, desc.head_dim
    _need(q, "q", desc.dtype, (layer_count, B, Hq, D))
    _need(k_new, "k_new", desc.dtype, (layer_count, B, H, D))
    _need(v_new, "v_new", desc.dtype, (layer_count, B, H, D))
    _need(out, "out", desc.dtype, (layer_count, B, Hq, D))
    _need(new_pos, "new_pos", torch.int32, (B,))
    _check_dense_state(desc, pc["score"], pc["pos"], pc["len"])
    d, ps = desc.c_struct(), _paged_struct(desc, pc)
    _check("voxzip_decode_step_paged", lib().voxzip_decode_step_paged(
        ctypes.byref(d), ctypes.byref(ps), int(layer_begin), int(layer_count), _ptr(q), _ptr(k_new), _ptr(v_new),
        _ptr(new_pos), _ptr(pc["score"]), _ptr(pc["pos"]), _ptr(pc["len"]), float(gamma), float(sm_scale),
        int(max_len), _ptr(out), _stream(stream)))


def voxzip_evict_paged(desc: CacheDesc, pc, layer_begin: int, layer_count: int, budget, *, sink: int = 4,
                       recent_frac: float = 0.2, history: bool = True, compaction: str = "ordered",
                       stream=None) -> None:
    """Eviction (Eq. 7-9, under a policy as voxzip_evict_ex) on a paged cache; the pages beyond the
    new length go back to the pool."""
    _check_dense_state(desc, pc["score"], pc["pos"], pc["len"])
    if budget.dim() == 1:
        _need(budget, "budget", torch.int32, (desc.batch,))
        sb, sl = 1, 0
    else:
        _need(budget, "budget", torch.int32, (desc.batch, desc.layers))
        sb, sl = desc.layers, 1
    if compaction not in ("ordered", "fill"):
        raise ValueError("compaction must be 'ordered' or 'fill'")
    pol = _EvictPolicy(int(sink), float(recent_frac), int(bool(history)), sb, sl,
                       VOXZIP_COMPACT_FILL if compaction == "fill" else VOXZIP_COMPACT_ORDERED)
    d, ps = desc.c_struct(), _paged_struct(desc, pc)
    _check("voxzip_evict_paged", lib().voxzip_evict_paged(
        ctypes.byref(d), ctypes.byref(ps), int(layer_begin), int(layer_count), _ptr(pc["score"]), _ptr(pc["pos"]),
        _ptr(pc["len"]), _ptr(budget), ctypes.byref(pol), _stream(stream)))


def voxzip_anchor_fuse_workspace_size(desc: CacheDesc, prefill_stride: int, num_spans: int) -> int:
    d = desc.c_struct()
    return int(lib().voxzip_anchor_fuse_workspace_size(ctypes.byref(d), int(prefill_stride), int(num_spans)))


def voxzip_anchor_fuse(desc: CacheDesc, k_prefill, v_prefill, in_len, audio_begin, audio_len, span_off,
                       span_start, span_end, span_groups, k_cache, v_cache, score, pos, len_, *,
                       slot_map=None, anchor_k=None, anchor_v=None, workspace=None, stream=None) -> None:
    """Stage 1 (Sec. 3.2.1): fuse the prefilled K/V of every unit into the cache."""
    B, L, H, D = desc.batch, desc.layers, desc.kv_heads, desc.head_dim
    if k_prefill.dim() != 5:
        raise ValueError("k_prefill must be [B][L][Hkv][stride][D]")
    stride = k_prefill.shape[3]
    _need(k_prefill, "k_prefill", desc.dtype, (B, L, H, stride, D), pinned_ok=True)
    _need(v_prefill, "v_prefill", desc.dtype, (B, L, H, stride, D), pinned_ok=True)
    for name, t in (("in_len", in_len), ("audio_begin", audio_begin), ("audio_len", audio_len)):
        _need(t, name, torch.int32, (B,))
    _need(span_off, "span_off", torch.int32, (B + 1,))
    num_spans = span_start.numel()
    for name, t in (("span_start", span_start), ("span_end", span_end), ("span_groups", span_groups)):
        _need(t, name, torch.int32, (num_spans,))
    _check_cache(desc, k_cache, v_cache, score, pos, len_)
    if slot_map is not None:
        _need(slot_map, "slot_map", torch.int32, (B, stride))
    anchor_stride = 0
    if anchor_k is not None or anchor_v is not None:
        anchor_stride = anchor_k.shape[3]
        _need(anchor_k, "anchor_k", desc.dtype, (B, L, H, anchor_stride, D))
        _need(anchor_v, "anchor_v", desc.dtype, (B, L, H, anchor_stride, D))
    need = voxzip_anchor_fuse_workspace_size(desc, stride, num_spans)
    if workspace is None:
        workspace = torch.empty(max(need, 256), dtype=torch.uint8, device=k_cache.device)
    _need(workspace, "workspace", torch.uint8)
    d = desc.c_struct()
    _check("voxzip_anchor_fuse", lib().voxzip_anchor_fuse(
        ctypes.byref(d), _ptr(k_prefill), _ptr(v_prefill), int(stride), _ptr(in_len), _ptr(audio_begin),
        _ptr(audio_len), _ptr(span_off), int(num_spans), _ptr(span_start), _ptr(span_end), _ptr(span_groups),
        _ptr(anchor_k), _ptr(anchor_v), int(anchor_stride), _ptr(k_cache), _ptr(v_cache), _ptr(score),
        _ptr(pos), _ptr(len_), _ptr(slot_map), _ptr(workspace), int(workspace.numel()), _stream(stream)))


def voxzip_segments_to_spans(t_start, t_end, confidence, text_len, tau_total: float, audio_len: int,
                             audio_begin: int = 0, threshold: float = 0.3) -> dict:
    """ASR segments -> token-index spans (host): the confidence filter and Eq. 3. Returns
    dict(start, end, groups, seg_index) of int32 numpy arrays, one entry per kept segment."""
    import numpy as np
    ts = np.ascontiguousarray(t_start, dtype=np.float64)
    te = np.ascontiguousarray(t_end, dtype=np.float64)
    cf = np.ascontiguousarray(confidence, dtype=np.float64)
    tl = np.ascontiguousarray(text_len, dtype=np.int32)
    n = len(ts)
    if not (len(te) == n and len(cf) == n and len(tl) == n):
        raise ValueError("t_start, t_end, confidence and text_len must have the same length")
    outs = [np.zeros(max(n, 1), np.int32) for _ in range(4)]
    k = ctypes.c_int32(0)
    p = lambda a: a.ctypes.data_as(ctypes.c_void_p)
    _check("voxzip_segments_to_spans", lib().voxzip_segments_to_spans(
        n, p(ts), p(te), p(cf), p(tl), float(tau_total), int(audio_len), int(audio_begin), float(threshold),
        *[p(a) for a in outs], ctypes.byref(k)))
    m = k.value
    return dict(start=outs[0][:m], end=outs[1][:m], groups=outs[2][:m], seg_index=outs[3][:m])


def voxzip_embed_fuse_workspace_size(desc: EmbedDesc, stride: int, num_spans: int) -> int:
    d = desc.c_struct()
    return int(lib().voxzip_embed_fuse_workspace_size(ctypes.byref(d), int(stride), int(num_spans)))


def voxzip_embed_fuse(desc: EmbedDesc, e_in, in_len, audio_begin, audio_len, span_off, span_start, span_end,
                      span_groups, e_out, pos, len_, *, e_text=None, keep_background: bool = True, slot_map=None,
                      workspace=None, stream=None) -> None:
    """Stage 1 at the embedding level (Sec. 3.2.1): fuse each sequence's audio embeddings under its
    semantic set, adding the embedded transcription as anchors; keep_background=False is the
    "Partial" configuration (uncovered audio dropped)."""
    B, D, C = desc.batch, desc.d_model, desc.capacity
    if e_in.dim() != 3:
        raise ValueError("e_in must be [B][stride][d_model]")
    stride = e_in.shape[1]
    _need(e_in, "e_in", desc.dtype, (B, stride, D))
    for name, t in (("in_len", in_len), ("audio_begin", audio_begin), ("audio_len", audio_len)):
        _need(t, name, torch.int32, (B,))
    _need(span_off, "span_off", torch.int32, (B + 1,))
    num_spans = span_start.numel()
    for name, t in (("span_start", span_start), ("span_end", span_end), ("span_groups", span_groups)):
        _need(t, name, torch.int32, (num_spans,))
    _need(e_out, "e_out", desc.dtype, (B, C, D))
    _need(pos, "pos", torch.int32, (B, C))
    _need(len_, "len", torch.int32, (B,))
    if slot_map is not None:
        _need(slot_map, "slot_map", torch.int32, (B, stride))
    text_stride = 0
    if e_text is not None:
        text_stride = e_text.shape[1]
        _need(e_text, "e_text", desc.dtype, (B, text_stride, D))
    need = voxzip_embed_fuse_workspace_size(desc, stride, num_spans)
    if workspace is None:
        workspace = torch.empty(max(need, 256), dtype=torch.uint8, device=e_out.device)
    _need(workspace, "workspace", torch.uint8)
    d = desc.c_struct()
    _check("voxzip_embed_fuse", lib().voxzip_embed_fuse(
        ctypes.byref(d), _ptr(e_in), int(stride), _ptr(in_len), _ptr(audio_begin), _ptr(audio_len), _ptr(span_off),
        int(num_spans), _ptr(span_start), _ptr(span_end), _ptr(span_groups), _ptr(e_text), int(text_stride),
        int(bool(keep_background)), _ptr(e_out), _ptr(pos), _ptr(len_), _ptr(slot_map), _ptr(workspace),
        int(workspace.numel()), _stream(stream)))


def voxzip_anchor_fuse_noalloc(desc: CacheDesc, k_prefill, v_prefill, in_len, audio_begin, audio_len, span_off,
                               span_start, span_end, span_groups, k_cache, v_cache, score, pos, len_, *,
                               slot_map=None, anchor_k=None, anchor_v=None, stream=None) -> None:
    """Stage 1 like voxzip_anchor_fuse, for callers that cannot allocate: the library's fixed
    4 MiB scratch replaces the workspace (VoxZipError with VOXZIP_ESCRATCH if it is too small)."""
    B, L, H, D = desc.batch, desc.layers, desc.kv_heads, desc.head_dim
    if k_prefill.dim() != 5:
        raise ValueError("k_prefill must be [B][L][Hkv][stride][D]")
    stride = k_prefill.shape[3]
    _need(k_prefill, "k_prefill", desc.dtype, (B, L, H, stride, D), pinned_ok=True)
    _need(v_prefill, "v_prefill", desc.dtype, (B, L, H, stride, D), pinned_ok=True)
    for name, t in (("in_len", in_len), ("audio_begin", audio_begin), ("audio_len", audio_len)):
        _need(t, name, torch.int32, (B,))
    _need(span_off, "span_off", torch.int32, (B + 1,))
    num_spans = span_start.numel()
    for name, t in (("span_start", span_start), ("span_end", span_end), ("span_groups", span_groups)):
        _need(t, name, torch.int32, (num_spans,))
    _check_cache(desc, k_cache, v_cache, score, pos, len_)
    if slot_map is not None:
        _need(slot_map, "slot_map", torch.int32, (B, stride))
    anchor_stride = 0
    if anchor_k is not None or anchor_v is not None:
        anchor_stride = anchor_k.shape[3]
        _need(anchor_k, "anchor_k", desc.dtype, (B, L, H, anchor_stride, D))
        _need(anchor_v, "anchor_v", desc.dtype, (B, L, H, anchor_stride, D))
    d = desc.c_struct()
    _check("voxzip_anchor_fuse_noalloc", lib().voxzip_anchor_fuse_noalloc(
        ctypes.byref(d), _ptr(k_prefill), _ptr(v_prefill), int(stride), _ptr(in_len), _ptr(audio_begin),
        _ptr(audio_len), _ptr(span_off), int(num_spans), _ptr(span_start), _ptr(span_end), _ptr(span_groups),
        _ptr(anchor_k), _ptr(anchor_v), int(anchor_stride), _ptr(k_cache), _ptr(v_cache), _ptr(score),
        _ptr(pos), _ptr(len_), _ptr(slot_map), _stream(stream)))


def voxzip_decode_step(desc: CacheDesc, layer_begin: int, layer_count: int, q, k_new, v_new, new_pos,
                       k_cache, v_cache, score, pos, len_, gamma: float, out, *, sm_scale: float = 0.0,
                       max_len: int = 0, stream=None) -> None:
    """One decode step (Eq. 1, Eq. 2, Eq. 6) for layers [layer_begin, layer_begin + layer_count)."""
    B, Hq, H, D = desc.batch, desc.q_heads, desc.kv_heads, desc.head_dim
    _need(q, "q", desc.dtype, (layer_count, B, Hq, D))
    _need(k_new, "k_new", desc.dtype, (layer_count, B, H, D))
    _need(v_new, "v_new", desc.dtype, (layer_count, B, H, D))
    _need(out, "out", desc.dtype, (layer_count, B, Hq, D))
    _need(new_pos, "new_pos", torch.int32, (B,))
    _check_cache(desc, k_cache, v_cache, score, pos, len_)
    d = desc.c_struct()
    _check("voxzip_decode_step", lib().voxzip_decode_step(
        ctypes.byref(d), int(layer_begin), int(layer_count), _ptr(q), _ptr(k_new), _ptr(v_new), _ptr(new_pos),
        _ptr(k_cache), _ptr(v_cache), _ptr(score), _ptr(pos), _ptr(len_), float(gamma), float(sm_scale),
        int(max_len), _ptr(out), _stream(stream)))


def voxzip_evict(desc: CacheDesc, layer_begin: int, layer_count: int, k_cache, v_cache, score, pos, len_,
                 budget, *, sink: int = 4, recent_frac: float = 0.2, stream=None) -> None:
    """Budgeted eviction (Eq. 7-9) for layers [layer_begin, layer_begin + layer_count)."""
    _check_cache(desc, k_cache, v_cache, score, pos, len_)
    _need(budget, "budget", torch.int32, (desc.batch,))
    d = desc.c_struct()
    _check("voxzip_evict", lib().voxzip_evict(
        ctypes.byref(d), int(layer_begin), int(layer_count), _ptr(k_cache), _ptr(v_cache), _ptr(score), _ptr(pos),
        _ptr(len_), _ptr(budget), int(sink), float(recent_frac), _stream(stream)))


def voxzip_evict_ex(desc: CacheDesc, layer_begin: int, layer_count: int, k_cache, v_cache, score, pos, len_,
                    budget, *, sink: int = 4, recent_frac: float = 0.2, history: bool = True,
                    compaction: str = "ordered", stream=None) -> None:
    """Eviction under a policy. `budget` is [B] (one per sequence) or [B][L] (one per layer);
    history=False is the StreamingLLM policy (sinks + a recent window of budget - sink rows);
    compaction="fill" chooses sinks / recents by position and fills the evicted slots with the kept
    rows beyond the budget (at most n - budget rows move)."""
    _check_cache(desc, k_cache, v_cache, score, pos, len_)
    if budget.dim() == 1:
        _need(budget, "budget", torch.int32, (desc.batch,))
        sb, sl = 1, 0
    else:
        _need(budget, "budget", torch.int32, (desc.batch, desc.layers))
        sb, sl = desc.layers, 1
    if compaction not in ("ordered", "fill"):
        raise ValueError("compaction must be 'ordered' or 'fill'")
    pol = _EvictPolicy(int(sink), float(recent_frac), int(bool(history)), sb, sl,
                       VOXZIP_COMPACT_FILL if compaction == "fill" else VOXZIP_COMPACT_ORDERED)
    d = desc.c_struct()
    _check("voxzip_evict_ex", lib().voxzip_evict_ex(
        ctypes.byref(d), int(layer_begin), int(layer_count), _ptr(k_cache), _ptr(v_cache), _ptr(score), _ptr(pos),
        _ptr(len_), _ptr(budget), ctypes.byref(pol), _stream(stream)))


def voxzip_selftest_bounded_wait(limit: int = 1000, stream=None) -> None:
    """Launches the bounded-wait self-test: a wait that can never complete gives up after `limit`
    polls and sets DEV_TIMEOUT in the status word (read it with voxzip_get_status)."""
    _check("voxzip_selftest_bounded_wait", lib().voxzip_selftest_bounded_wait(int(limit), _stream(stream)))


def voxzip_stream_read(buf: torch.Tensor, nbytes: int, sink: torch.Tensor, stream=None) -> None:
    """Measurement helper: one plain streaming read of the first `nbytes` of `buf` (a multiple of 16),
    launched like the decode step; `sink` is a one-element int32 device tensor."""
    if not buf.is_cuda or nbytes > buf.numel() * buf.element_size():
        raise ValueError("buf must be a device tensor of at least nbytes")
    _need(sink, "sink", torch.int32)
    _check("voxzip_stream_read", lib().voxzip_stream_read(_ptr(buf), int(nbytes), _ptr(sink), _stream(stream)))


def voxzip_get_status(stream=None) -> int:
    """Waits for the stream, then returns and clears the device status word (DEV_* bits)."""
    bits = ctypes.c_uint32(0)
    _check("voxzip_get_status", lib().voxzip_get_status(ctypes.byref(bits), _stream(stream)))
    return int(bits.value)
