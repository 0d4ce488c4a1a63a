"""VoxZip KV-cache compression for GB300 (sm_103a): a C-ABI CUDA library and its Python binding.

The three steps of the path (arxiv 2608.08569, Sec. 3.2):
  voxzip_anchor_fuse   stage-1 semantic-anchored fusion of the prefilled cache (Eq. 4-5)
  voxzip_decode_step   append + GQA attention + decayed accumulated score (Eq. 1, 2, 6)
  voxzip_evict         sinks + recent window + top-N history, compacted in place (Eq. 7-9)
  voxzip_evict_ex      the same under a policy: per-layer budgets, no history (StreamingLLM),
                       hole-filling compaction (at most n - budget rows move)
Paged cache (pages of 64 rows, a device-side free stack; memory follows the live cache):
  allocate_paged_cache, voxzip_paged_init, voxzip_anchor_fuse_paged, voxzip_decode_step_paged,
  voxzip_evict_paged
Stage 1 where the paper runs it, on input embeddings from ASR output:
  voxzip_segments_to_spans   confidence filter + time-to-index map (Eq. 3), on the host
  voxzip_embed_fuse          the same fusion on [B][tokens][d_model] embeddings with text anchors
"""
from ._native import (CacheDesc, EmbedDesc, VoxZipError, allocate_cache, lib, voxzip_anchor_fuse,
                      voxzip_anchor_fuse_noalloc, voxzip_anchor_fuse_workspace_size, voxzip_decode_step,
                      voxzip_embed_fuse, voxzip_embed_fuse_workspace_size, voxzip_evict, voxzip_evict_ex,
                      voxzip_get_status, voxzip_segments_to_spans)
from ._native import (voxzip_selftest_bounded_wait, voxzip_stream_read)
from ._native import (PAGE_TOKENS, allocate_paged_cache, paged_pages_in_use, voxzip_anchor_fuse_paged,
                      voxzip_decode_step_paged, voxzip_evict_paged, voxzip_paged_init)
from ._native import (DEV_BAD_BUDGET, DEV_BAD_POSITIONS, DEV_BOUNDS, DEV_BAD_SPANS, DEV_CAPACITY, DEV_LEN_HINT, DEV_TIMEOUT, VOXZIP_ECUDA,
                      VOXZIP_EINVAL, VOXZIP_ESCRATCH, VOXZIP_EUNSUPPORTED, VOXZIP_OK)

__all__ = ["voxzip_selftest_bounded_wait", "voxzip_stream_read", "PAGE_TOKENS", "allocate_paged_cache", "paged_pages_in_use", "voxzip_anchor_fuse_paged",
           "voxzip_decode_step_paged", "voxzip_evict_paged", "voxzip_paged_init", "CacheDesc", "EmbedDesc", "voxzip_evict_ex", "DEV_BAD_POSITIONS", "DEV_BOUNDS", "voxzip_embed_fuse", "voxzip_embed_fuse_workspace_size",
           "voxzip_segments_to_spans", "VoxZipError", "allocate_cache", "lib", "voxzip_anchor_fuse", "voxzip_anchor_fuse_noalloc",
           "voxzip_anchor_fuse_workspace_size", "voxzip_decode_step", "voxzip_evict", "voxzip_get_status",
           "DEV_BAD_BUDGET", "DEV_BAD_SPANS", "DEV_CAPACITY", "DEV_LEN_HINT", "DEV_TIMEOUT", "VOXZIP_ECUDA",
           "VOXZIP_EINVAL", "VOXZIP_ESCRATCH", "VOXZIP_EUNSUPPORTED", "VOXZIP_OK"]
