// Paged K/V storage: slot s of unit u is row (s % 64) of page table[u][s / 64] of a pool. The
// free pages are a device-side stack (an array and a count), so pages are taken and returned
// inside the kernels of the decode loop.
#pragma once

#include <cuda_runtime.h>
#include <stddef.h>
#include <stdint.h>

#include "voxzip.h"

namespace voxzip {

constexpr int kPageTokens = VOXZIP_PAGE_TOKENS;
static_assert(kPageTokens == 64, "page = one 64-token tile of the decode kernel");

struct PageView {
    int32_t *table;       // [units][max_pages]
    int32_t *free_pages;  // [pages]
    int32_t *free_count;
    int32_t max_pages;
};

// Row of the pool that holds slot s of cache unit cu (the page must exist).
__device__ __forceinline__ int64_t paged_row(const PageView &pv, int64_t cu, int32_t s) {
    return (int64_t)pv.table[cu * pv.max_pages + (s >> 6)] * kPageTokens + (s & (kPageTokens - 1));
}

// Takes one free page, or returns -1 when none is left.
__device__ __forceinline__ int32_t take_page(const PageView &pv) {
    const int32_t t = atomicSub(pv.free_count, 1);
    if (t <= 0) {
        atomicAdd(pv.free_count, 1);
        return -1;
    }
    return pv.free_pages[t - 1];
}

// Returns the pages of unit cu with page index in [p0, p1) to the stack (one warp, all lanes).
__device__ __forceinline__ void return_pages_warp(const PageView &pv, int64_t cu, int32_t p0, int32_t p1) {
    const int lane = threadIdx.x & 31;
    int32_t *row = pv.table + cu * pv.max_pages;
    for (int32_t base = p0; base < p1; base += 32) {
        const int32_t p = base + lane;
        const int32_t page = p < p1 ? row[p] : -1;
        const unsigned have = __ballot_sync(0xffffffffu, page >= 0);
        int32_t at = 0;
        if (lane == 0 && have) at = atomicAdd(pv.free_count, __popc(have));
        at = __shfl_sync(0xffffffffu, at, 0);
        if (page >= 0) {
            pv.free_pages[at + __popc(have & ((1u << lane) - 1u))] = page;
            row[p] = -1;
        }
    }
}

cudaError_t launch_paged_init(const voxzip_cache_desc &d, const voxzip_paged_cache &pc, int32_t *len,
                              cudaStream_t stream);

size_t anchor_fuse_paged_workspace_bytes(const voxzip_cache_desc &d, int32_t prefill_stride, int32_t num_spans);

cudaError_t launch_anchor_fuse_paged(const voxzip_cache_desc &d, const voxzip_paged_cache &pc, const void *k_prefill,
                                     const void *v_prefill, int32_t prefill_stride, const int32_t *in_len,
                                     const int32_t *audio_begin, const int32_t *audio_len, const int32_t *span_off,
                                     int32_t num_spans, const int32_t *span_start, const int32_t *span_end,
                                     const int32_t *span_groups, const void *anchor_k, const void *anchor_v,
                                     int32_t anchor_stride, float *score, int32_t *pos, int32_t *len,
                                     int32_t *slot_map, void *workspace, int32_t *status, cudaStream_t stream);

bool decode_mma_paged_supported(const voxzip_cache_desc &d);

cudaError_t launch_decode_mma_paged(const voxzip_cache_desc &d, const voxzip_paged_cache &pc, int32_t layer_begin,
                                    int32_t layer_count, const void *q, const void *k_new, const void *v_new,
                                    const int32_t *new_pos, float *score, int32_t *pos, int32_t *len, float gamma,
                                    float sm_scale, int32_t max_len, void *out, int32_t *status, cudaStream_t stream,
                                    bool *unsupported);

cudaError_t launch_evict_paged(const voxzip_cache_desc &d, const voxzip_paged_cache &pc, int32_t layer_begin,
                               int32_t layer_count, float *score, int32_t *pos, int32_t *len, const int32_t *budget,
                               const voxzip_evict_policy &policy, int32_t *status, cudaStream_t stream);

}  // namespace voxzip
