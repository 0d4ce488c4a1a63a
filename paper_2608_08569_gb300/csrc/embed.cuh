// Launchers of the embedding-level stage 1 (anchor_fuse.cu), called by the C ABI (api.cu).
#pragma once

#include <cuda_runtime.h>
#include <stddef.h>
#include <stdint.h>

namespace voxzip {

size_t embed_fuse_workspace_bytes(int32_t batch, int32_t stride, int32_t num_spans);

cudaError_t launch_embed_fuse(int32_t B, int32_t D, int32_t C, bool bf16, const void *e_in, int32_t stride,
                              const int32_t *in_len, const int32_t *audio_begin, const int32_t *audio_len,
                              const int32_t *span_off, int32_t num_spans, const int32_t *span_start,
                              const int32_t *span_end, const int32_t *span_groups, const void *e_text,
                              int32_t text_stride, bool keep_background, void *e_out, int32_t *pos, int32_t *len,
                              int32_t *slot_map, void *workspace, int32_t *status, cudaStream_t stream);

}  // namespace voxzip
