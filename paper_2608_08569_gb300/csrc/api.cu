// C ABI of the VoxZip library (declared in include/voxzip.h): argument validation, the device
// status word, and dispatch to the kernel launchers. Nothing here allocates device memory. Every
// entry point opens an NVTX range of its own name (a no-op unless a profiler listens).
#include <math.h>

#include <atomic>
#include <nvtx3/nvToolsExt.h>

#include "common.cuh"
#include "embed.cuh"
#include "evict_policy.cuh"
#include "paged.cuh"
#include "ptx.cuh"

namespace {

// Asynchronous error bits (VOXZIP_DEV_*) raised by the kernels of this library on this device.
__device__ int32_t g_status_word;

constexpr int kMaxDevices = 64;
// Device address of g_status_word, per device. Host threads may make their first call on a device
// at the same time: each looks the address up and stores the same value, so atomics make that race
// well defined without a lock.
std::atomic<int32_t *> g_status_addr[kMaxDevices];

// Address of the status word on the current device (looked up once per device).
voxzip_status status_word(int32_t **addr) {
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return VOXZIP_ECUDA;
    int32_t *a = g_status_addr[dev].load(std::memory_order_acquire);
    if (a == nullptr) {
        void *p = nullptr;
        if (cudaGetSymbolAddress(&p, g_status_word) != cudaSuccess) return VOXZIP_ECUDA;
        a = static_cast<int32_t *>(p);
        g_status_addr[dev].store(a, std::memory_order_release);
    }
    *addr = a;
    return VOXZIP_OK;
}

bool desc_ok(const voxzip_cache_desc *d) {
    if (d == nullptr) return false;
    if (d->batch < 1 || d->layers < 1 || d->q_heads < 1 || d->kv_heads < 1 || d->capacity < 1) return false;
    if (d->q_heads % d->kv_heads != 0) return false;
    if (d->head_dim != 64 && d->head_dim != 128) return false;
    if (d->dtype != VOXZIP_F32 && d->dtype != VOXZIP_BF16) return false;
    // element counts of the largest tensors must fit int64 and slot indices int32
    const int64_t units = (int64_t)d->batch * d->layers * d->kv_heads;
    if (units > (int64_t)1 << 31) return false;
    return true;
}

bool aligned16(const void *p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

voxzip_status from_cuda(cudaError_t e) { return e == cudaSuccess ? VOXZIP_OK : VOXZIP_ECUDA; }

constexpr int kMaxGridY = 65535;

// An NVTX range for the lifetime of an entry point.
struct Range {
    explicit Range(const char *name) { nvtxRangePushA(name); }
    ~Range() { nvtxRangePop(); }
};

// One CTA: an mbarrier armed for 16 bytes that never arrive, waited on with the bounded wait.
__global__ void selftest_wait_kernel(uint32_t limit, int32_t *status) {
    __shared__ uint64_t bar;
    if (threadIdx.x == 0) {
        voxzip::ptx::mbar_init(&bar, 1);
        voxzip::ptx::fence_mbar_init();
        voxzip::ptx::mbar_arrive_expect_tx(&bar, 16);
        if (!voxzip::ptx::mbar_wait_bounded(&bar, 0, limit)) voxzip::raise_status(status, VOXZIP_DEV_TIMEOUT);
    }
}

}  // namespace

// The status word's device address on the current device, for entry points in other files.
voxzip_status voxzip_status_word_address(int32_t **addr) { return status_word(addr); }

extern "C" {

int32_t voxzip_version(void) { return 100; }

const char *voxzip_status_string(voxzip_status s) {
    switch (s) {
        case VOXZIP_OK: return "VOXZIP_OK";
        case VOXZIP_EINVAL: return "VOXZIP_EINVAL";
        case VOXZIP_EUNSUPPORTED: return "VOXZIP_EUNSUPPORTED";
        case VOXZIP_ECUDA: return "VOXZIP_ECUDA";
        case VOXZIP_ESCRATCH: return "VOXZIP_ESCRATCH";
    }
    return "VOXZIP_UNKNOWN";
}

size_t voxzip_anchor_fuse_workspace_size(const voxzip_cache_desc *desc, int32_t prefill_stride,
                                         int32_t num_spans) {
    Range range("voxzip_anchor_fuse_workspace_size");
    if (!desc_ok(desc) || prefill_stride < 1 || num_spans < 0) return 0;
    return voxzip::anchor_fuse_workspace_bytes(*desc, prefill_stride, num_spans);
}

voxzip_status voxzip_anchor_fuse(const voxzip_cache_desc *desc, const void *k_prefill,
                                 const void *v_prefill, int32_t prefill_stride,
                                 const int32_t *in_len, const int32_t *audio_begin,
                                 const int32_t *audio_len, const int32_t *span_off,
                                 int32_t num_spans, const int32_t *span_start,
                                 const int32_t *span_end, const int32_t *span_groups,
                                 const void *anchor_k, const void *anchor_v, int32_t anchor_stride,
                                 void *k_cache, void *v_cache, float *score, int32_t *pos,
                                 int32_t *len, int32_t *slot_map, void *workspace,
                                 size_t workspace_bytes, voxzip_stream_t stream) {
    Range range("voxzip_anchor_fuse");
    if (!desc_ok(desc) || prefill_stride < 1 || num_spans < 0) return VOXZIP_EINVAL;
    if (!k_prefill || !v_prefill || !in_len || !audio_begin || !audio_len || !span_off || !k_cache ||
        !v_cache || !score || !pos || !len || !workspace)
        return VOXZIP_EINVAL;
    if (num_spans > 0 && (!span_start || !span_end || !span_groups)) return VOXZIP_EINVAL;
    if ((anchor_k == nullptr) != (anchor_v == nullptr)) return VOXZIP_EINVAL;
    if (anchor_k && anchor_stride < 1) return VOXZIP_EINVAL;
    if (!aligned16(k_prefill) || !aligned16(v_prefill) || !aligned16(k_cache) || !aligned16(v_cache) ||
        (anchor_k && (!aligned16(anchor_k) || !aligned16(anchor_v))))
        return VOXZIP_EINVAL;
    if ((reinterpret_cast<uintptr_t>(workspace) & 255u) != 0) return VOXZIP_EINVAL;
    if (workspace_bytes < voxzip::anchor_fuse_workspace_bytes(*desc, prefill_stride, num_spans))
        return VOXZIP_EINVAL;
    if ((int64_t)desc->batch * desc->layers * desc->kv_heads > kMaxGridY || desc->batch > kMaxGridY)
        return VOXZIP_EUNSUPPORTED;
    int32_t *status = nullptr;
    voxzip_status st = status_word(&status);
    if (st != VOXZIP_OK) return st;
    return from_cuda(voxzip::launch_anchor_fuse(
        *desc, k_prefill, v_prefill, prefill_stride, in_len, audio_begin, audio_len, span_off, num_spans,
        span_start, span_end, span_groups, anchor_k, anchor_v, anchor_stride, k_cache, v_cache, score, pos, len,
        slot_map, workspace, status, reinterpret_cast<cudaStream_t>(stream)));
}

namespace {
bool paged_ok(const voxzip_cache_desc *d, const voxzip_paged_cache *pc) {
    if (!desc_ok(d) || pc == nullptr) return false;
    if (!pc->k_pool || !pc->v_pool || !pc->page_table || !pc->free_pages || !pc->free_count) return false;
    if (!aligned16(pc->k_pool) || !aligned16(pc->v_pool)) return false;
    const int64_t units = (int64_t)d->batch * d->layers * d->kv_heads;
    if (pc->max_pages < 1 || (int64_t)pc->max_pages * VOXZIP_PAGE_TOKENS != d->capacity) return false;
    if (pc->pages < units || (int64_t)pc->pages * VOXZIP_PAGE_TOKENS > INT32_MAX) return false;
    return true;
}

bool policy_ok(const voxzip_evict_policy &p) {
    if (p.sink < 0 || !(p.recent_frac >= 0.f && p.recent_frac <= 1.f)) return false;
    if ((p.history != 0 && p.history != 1) || p.budget_stride_b < 0 || p.budget_stride_l < 0) return false;
    return p.compaction == VOXZIP_COMPACT_ORDERED || p.compaction == VOXZIP_COMPACT_FILL;
}
}  // namespace

voxzip_status voxzip_paged_init(const voxzip_cache_desc *desc, const voxzip_paged_cache *paged, int32_t *len,
                                voxzip_stream_t stream) {
    Range range("voxzip_paged_init");
    if (!paged_ok(desc, paged) || !len) return VOXZIP_EINVAL;
    return from_cuda(voxzip::launch_paged_init(*desc, *paged, len, reinterpret_cast<cudaStream_t>(stream)));
}

size_t voxzip_anchor_fuse_paged_workspace_size(const voxzip_cache_desc *desc, int32_t prefill_stride,
                                               int32_t num_spans) {
    Range range("voxzip_anchor_fuse_paged_workspace_size");
    if (!desc_ok(desc) || prefill_stride < 1 || num_spans < 0) return 0;
    return voxzip::anchor_fuse_paged_workspace_bytes(*desc, prefill_stride, num_spans);
}

voxzip_status voxzip_anchor_fuse_paged(const voxzip_cache_desc *desc, const voxzip_paged_cache *paged,
                                       const void *k_prefill, const void *v_prefill,
                                       int32_t prefill_stride, const int32_t *in_len,
                                       const int32_t *audio_begin, const int32_t *audio_len,
                                       const int32_t *span_off, int32_t num_spans,
                                       const int32_t *span_start, const int32_t *span_end,
                                       const int32_t *span_groups, const void *anchor_k,
                                       const void *anchor_v, int32_t anchor_stride, float *score,
                                       int32_t *pos, int32_t *len, int32_t *slot_map, void *workspace,
                                       size_t workspace_bytes, voxzip_stream_t stream) {
    Range range("voxzip_anchor_fuse_paged");
    if (!paged_ok(desc, paged) || prefill_stride < 1 || num_spans < 0) return VOXZIP_EINVAL;
    if (!k_prefill || !v_prefill || !in_len || !audio_begin || !audio_len || !span_off || !score || !pos || !len ||
        !workspace)
        return VOXZIP_EINVAL;
    if (num_spans > 0 && (!span_start || !span_end || !span_groups)) return VOXZIP_EINVAL;
    if ((anchor_k == nullptr) != (anchor_v == nullptr)) return VOXZIP_EINVAL;
    if (anchor_k && anchor_stride < 1) return VOXZIP_EINVAL;
    if (!aligned16(k_prefill) || !aligned16(v_prefill) || (anchor_k && (!aligned16(anchor_k) || !aligned16(anchor_v))))
        return VOXZIP_EINVAL;
    if ((reinterpret_cast<uintptr_t>(workspace) & 255u) != 0) return VOXZIP_EINVAL;
    if (workspace_bytes < voxzip::anchor_fuse_paged_workspace_bytes(*desc, prefill_stride, num_spans))
        return VOXZIP_EINVAL;
    if ((int64_t)desc->batch * desc->layers * desc->kv_heads > kMaxGridY || desc->batch > kMaxGridY)
        return VOXZIP_EUNSUPPORTED;
    int32_t *status = nullptr;
    voxzip_status st = status_word(&status);
    if (st != VOXZIP_OK) return st;
    return from_cuda(voxzip::launch_anchor_fuse_paged(
        *desc, *paged, k_prefill, v_prefill, prefill_stride, in_len, audio_begin, audio_len, span_off, num_spans,
        span_start, span_end, span_groups, anchor_k, anchor_v, anchor_stride, score, pos, len, slot_map, workspace,
        status, reinterpret_cast<cudaStream_t>(stream)));
}

voxzip_status voxzip_decode_step_paged(const voxzip_cache_desc *desc, const voxzip_paged_cache *paged,
                                       int32_t layer_begin, int32_t layer_count, const void *q,
                                       const void *k_new, const void *v_new, const int32_t *new_pos,
                                       float *score, int32_t *pos, int32_t *len, float gamma,
                                       float sm_scale, int32_t max_len, void *out,
                                       voxzip_stream_t stream) {
    Range range("voxzip_decode_step_paged");
    if (!paged_ok(desc, paged)) return VOXZIP_EINVAL;
    if (layer_begin < 0 || layer_count < 1 || layer_begin + (int64_t)layer_count > desc->layers)
        return VOXZIP_EINVAL;
    if (!q || !k_new || !v_new || !new_pos || !score || !pos || !len || !out) return VOXZIP_EINVAL;
    if (!(gamma > 0.f && gamma <= 1.f) || isnan(sm_scale) || isinf(sm_scale)) return VOXZIP_EINVAL;
    if (!aligned16(q) || !aligned16(k_new) || !aligned16(v_new) || !aligned16(out)) return VOXZIP_EINVAL;
    if (!voxzip::decode_mma_paged_supported(*desc)) return VOXZIP_EUNSUPPORTED;
    if ((int64_t)layer_count * desc->batch * desc->kv_heads > kMaxGridY) return VOXZIP_EUNSUPPORTED;
    int32_t *status = nullptr;
    voxzip_status st = status_word(&status);
    if (st != VOXZIP_OK) return st;
    bool unsupported = false;
    cudaError_t e = voxzip::launch_decode_mma_paged(*desc, *paged, layer_begin, layer_count, q, k_new, v_new, new_pos,
                                                    score, pos, len, gamma, sm_scale, max_len, out, status,
                                                    reinterpret_cast<cudaStream_t>(stream), &unsupported);
    if (unsupported) return VOXZIP_EUNSUPPORTED;
    return from_cuda(e);
}

voxzip_status voxzip_evict_paged(const voxzip_cache_desc *desc, const voxzip_paged_cache *paged,
                                 int32_t layer_begin, int32_t layer_count, float *score, int32_t *pos,
                                 int32_t *len, const int32_t *budget, const voxzip_evict_policy *policy,
                                 voxzip_stream_t stream) {
    Range range("voxzip_evict_paged");
    if (!paged_ok(desc, paged) || policy == nullptr || !policy_ok(*policy)) return VOXZIP_EINVAL;
    if (layer_begin < 0 || layer_count < 1 || layer_begin + (int64_t)layer_count > desc->layers)
        return VOXZIP_EINVAL;
    if (!score || !pos || !len || !budget) return VOXZIP_EINVAL;
    if ((int64_t)layer_count * desc->batch * desc->kv_heads > ((int64_t)1 << 31) - 1) return VOXZIP_EUNSUPPORTED;
    int32_t *status = nullptr;
    voxzip_status st = status_word(&status);
    if (st != VOXZIP_OK) return st;
    return from_cuda(voxzip::launch_evict_paged(*desc, *paged, layer_begin, layer_count, score, pos, len, budget,
                                                *policy, status, reinterpret_cast<cudaStream_t>(stream)));
}

voxzip_status voxzip_segments_to_spans(int32_t n, const double *t_start, const double *t_end,
                                       const double *confidence, const int32_t *text_len,
                                       double tau_total, int32_t audio_len, int32_t audio_begin,
                                       double threshold, int32_t *span_start, int32_t *span_end,
                                       int32_t *span_groups, int32_t *seg_index,
                                       int32_t *num_spans) {
    Range range("voxzip_segments_to_spans");
    if (n < 0 || !num_spans || !(tau_total > 0.0) || isinf(tau_total) || audio_len < 0 || audio_begin < 0 ||
        (int64_t)audio_begin + audio_len > INT32_MAX)
        return VOXZIP_EINVAL;
    if (n > 0 && (!t_start || !t_end || !confidence || !text_len || !span_start || !span_end || !span_groups ||
                  !seg_index))
        return VOXZIP_EINVAL;
    for (int32_t i = 0; i < n; ++i)
        if (!(t_end[i] >= t_start[i]) || text_len[i] < 1 || (i > 0 && !(t_start[i] >= t_start[i - 1])))
            return VOXZIP_EINVAL;
    // Eq. 3 on one time: floor(L_a * (t / tau_total)) clamped to the audio.
    auto index_of = [&](double t) -> int64_t {
        const double f = floor((double)audio_len * (t / tau_total));
        if (!(f > 0.0)) return 0;  // also NaN
        return f >= (double)audio_len ? audio_len : (int64_t)f;
    };
    int32_t out = 0;
    int64_t end_prev = 0;
    for (int32_t i = 0; i < n; ++i) {
        if (!(confidence[i] > threshold)) continue;  // the confidence filter
        int64_t a = index_of(t_start[i]), b = index_of(t_end[i]);
        a = a < end_prev ? end_prev : a;
        b = b < a ? a : b;
        span_start[out] = (int32_t)(audio_begin + a);
        span_end[out] = (int32_t)(audio_begin + b);
        span_groups[out] = text_len[i];
        seg_index[out] = i;
        end_prev = b;
        ++out;
    }
    *num_spans = out;
    return VOXZIP_OK;
}

namespace {
bool embed_desc_ok(const voxzip_embed_desc *d) {
    if (d == nullptr || d->batch < 1 || d->d_model < 1 || d->capacity < 1) return false;
    if (d->dtype != VOXZIP_F32 && d->dtype != VOXZIP_BF16) return false;
    const int elems16 = d->dtype == VOXZIP_BF16 ? 8 : 4;  // elements per 16-byte vector
    return d->d_model % elems16 == 0;
}
}  // namespace

size_t voxzip_embed_fuse_workspace_size(const voxzip_embed_desc *desc, int32_t stride, int32_t num_spans) {
    Range range("voxzip_embed_fuse_workspace_size");
    if (!embed_desc_ok(desc) || stride < 1 || num_spans < 0) return 0;
    return voxzip::embed_fuse_workspace_bytes(desc->batch, stride, num_spans);
}

voxzip_status voxzip_embed_fuse(const voxzip_embed_desc *desc, const void *e_in, int32_t stride,
                                const int32_t *in_len, const int32_t *audio_begin,
                                const int32_t *audio_len, const int32_t *span_off,
                                int32_t num_spans, const int32_t *span_start,
                                const int32_t *span_end, const int32_t *span_groups,
                                const void *e_text, int32_t text_stride, int32_t keep_background,
                                void *e_out, int32_t *pos, int32_t *len, int32_t *slot_map,
                                void *workspace, size_t workspace_bytes, voxzip_stream_t stream) {
    Range range("voxzip_embed_fuse");
    if (!embed_desc_ok(desc) || stride < 1 || num_spans < 0) return VOXZIP_EINVAL;
    if (!e_in || !in_len || !audio_begin || !audio_len || !span_off || !e_out || !pos || !len || !workspace)
        return VOXZIP_EINVAL;
    if (num_spans > 0 && (!span_start || !span_end || !span_groups)) return VOXZIP_EINVAL;
    if (e_text && text_stride < 1) return VOXZIP_EINVAL;
    if (keep_background != 0 && keep_background != 1) return VOXZIP_EINVAL;
    if (!aligned16(e_in) || !aligned16(e_out) || (e_text && !aligned16(e_text))) return VOXZIP_EINVAL;
    if ((reinterpret_cast<uintptr_t>(workspace) & 255u) != 0) return VOXZIP_EINVAL;
    if (workspace_bytes < voxzip::embed_fuse_workspace_bytes(desc->batch, stride, num_spans)) return VOXZIP_EINVAL;
    if (desc->batch > kMaxGridY) return VOXZIP_EUNSUPPORTED;
    int32_t *status = nullptr;
    voxzip_status st = status_word(&status);
    if (st != VOXZIP_OK) return st;
    return from_cuda(voxzip::launch_embed_fuse(desc->batch, desc->d_model, desc->capacity,
                                               desc->dtype == VOXZIP_BF16, e_in, stride, in_len, audio_begin,
                                               audio_len, span_off, num_spans, span_start, span_end, span_groups,
                                               e_text, text_stride, keep_background != 0, e_out, pos, len, slot_map,
                                               workspace, status, reinterpret_cast<cudaStream_t>(stream)));
}

voxzip_status voxzip_decode_step(const voxzip_cache_desc *desc, int32_t layer_begin,
                                 int32_t layer_count, const void *q, const void *k_new,
                                 const void *v_new, const int32_t *new_pos, void *k_cache,
                                 void *v_cache, float *score, int32_t *pos, int32_t *len,
                                 float gamma, float sm_scale, int32_t max_len, void *out,
                                 voxzip_stream_t stream) {
    Range range("voxzip_decode_step");
    if (!desc_ok(desc)) return VOXZIP_EINVAL;
    if (layer_begin < 0 || layer_count < 1 || layer_begin + (int64_t)layer_count > desc->layers)
        return VOXZIP_EINVAL;
    if (!q || !k_new || !v_new || !new_pos || !k_cache || !v_cache || !score || !pos || !len || !out)
        return VOXZIP_EINVAL;
    if (!(gamma > 0.f && gamma <= 1.f) || isnan(sm_scale) || isinf(sm_scale)) return VOXZIP_EINVAL;
    if (!aligned16(q) || !aligned16(k_new) || !aligned16(v_new) || !aligned16(k_cache) || !aligned16(v_cache) ||
        !aligned16(out))
        return VOXZIP_EINVAL;
    if (desc->q_heads / desc->kv_heads > voxzip::kMaxGroup) return VOXZIP_EUNSUPPORTED;
    if ((int64_t)layer_count * desc->batch * desc->kv_heads > kMaxGridY) return VOXZIP_EUNSUPPORTED;
    int32_t *status = nullptr;
    voxzip_status st = status_word(&status);
    if (st != VOXZIP_OK) return st;
    bool unsupported = false;
    cudaError_t e = voxzip::launch_decode(*desc, layer_begin, layer_count, q, k_new, v_new, new_pos, k_cache,
                                          v_cache, score, pos, len, gamma, sm_scale, max_len, out, status,
                                          reinterpret_cast<cudaStream_t>(stream), &unsupported);
    if (unsupported) return VOXZIP_EUNSUPPORTED;
    return from_cuda(e);
}

voxzip_status voxzip_evict(const voxzip_cache_desc *desc, int32_t layer_begin,
                           int32_t layer_count, void *k_cache, void *v_cache, float *score,
                           int32_t *pos, int32_t *len, const int32_t *budget, int32_t sink,
                           float recent_frac, voxzip_stream_t stream) {
    Range range("voxzip_evict");
    if (!desc_ok(desc)) return VOXZIP_EINVAL;
    if (layer_begin < 0 || layer_count < 1 || layer_begin + (int64_t)layer_count > desc->layers)
        return VOXZIP_EINVAL;
    if (!k_cache || !v_cache || !score || !pos || !len || !budget) return VOXZIP_EINVAL;
    if (sink < 0 || !(recent_frac >= 0.f && recent_frac <= 1.f)) return VOXZIP_EINVAL;
    if (!aligned16(k_cache) || !aligned16(v_cache)) return VOXZIP_EINVAL;
    if ((int64_t)layer_count * desc->batch * desc->kv_heads > ((int64_t)1 << 31) - 1) return VOXZIP_EUNSUPPORTED;
    int32_t *status = nullptr;
    voxzip_status st = status_word(&status);
    if (st != VOXZIP_OK) return st;
    return from_cuda(voxzip::launch_evict(*desc, layer_begin, layer_count, k_cache, v_cache, score, pos, len,
                                          budget, sink, recent_frac, status,
                                          reinterpret_cast<cudaStream_t>(stream)));
}

voxzip_status voxzip_evict_ex(const voxzip_cache_desc *desc, int32_t layer_begin,
                              int32_t layer_count, void *k_cache, void *v_cache, float *score,
                              int32_t *pos, int32_t *len, const int32_t *budget,
                              const voxzip_evict_policy *policy, voxzip_stream_t stream) {
    Range range("voxzip_evict_ex");
    if (!desc_ok(desc) || policy == nullptr) return VOXZIP_EINVAL;
    if (layer_begin < 0 || layer_count < 1 || layer_begin + (int64_t)layer_count > desc->layers)
        return VOXZIP_EINVAL;
    if (!k_cache || !v_cache || !score || !pos || !len || !budget) return VOXZIP_EINVAL;
    const voxzip_evict_policy &p = *policy;
    if (p.sink < 0 || !(p.recent_frac >= 0.f && p.recent_frac <= 1.f)) return VOXZIP_EINVAL;
    if ((p.history != 0 && p.history != 1) || p.budget_stride_b < 0 || p.budget_stride_l < 0) return VOXZIP_EINVAL;
    if (p.compaction != VOXZIP_COMPACT_ORDERED && p.compaction != VOXZIP_COMPACT_FILL) return VOXZIP_EINVAL;
    if (!aligned16(k_cache) || !aligned16(v_cache)) return VOXZIP_EINVAL;
    if ((int64_t)layer_count * desc->batch * desc->kv_heads > ((int64_t)1 << 31) - 1) return VOXZIP_EUNSUPPORTED;
    int32_t *status = nullptr;
    voxzip_status st = status_word(&status);
    if (st != VOXZIP_OK) return st;
    return from_cuda(voxzip::launch_evict_policy(*desc, layer_begin, layer_count, k_cache, v_cache, score, pos,
                                                 len, budget, p, status, reinterpret_cast<cudaStream_t>(stream)));
}

voxzip_status voxzip_get_status(uint32_t *bits, voxzip_stream_t stream) {
    Range range("voxzip_get_status");
    if (!bits) return VOXZIP_EINVAL;
    int32_t *status = nullptr;
    voxzip_status st = status_word(&status);
    if (st != VOXZIP_OK) return st;
    cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
    int32_t host = 0;
    if (cudaStreamSynchronize(s) != cudaSuccess) return VOXZIP_ECUDA;
    if (cudaMemcpyAsync(&host, status, sizeof(int32_t), cudaMemcpyDeviceToHost, s) != cudaSuccess)
        return VOXZIP_ECUDA;
    if (cudaMemsetAsync(status, 0, sizeof(int32_t), s) != cudaSuccess) return VOXZIP_ECUDA;
    if (cudaStreamSynchronize(s) != cudaSuccess) return VOXZIP_ECUDA;
    *bits = (uint32_t)host;
    return VOXZIP_OK;
}

}  // extern "C"

extern "C" voxzip_status voxzip_selftest_bounded_wait(uint32_t limit, voxzip_stream_t stream) {
    Range range("voxzip_selftest_bounded_wait");
    if (limit < 1 || limit > (1u << 20)) return VOXZIP_EINVAL;
    int32_t *status = nullptr;
    voxzip_status st = status_word(&status);
    if (st != VOXZIP_OK) return st;
    selftest_wait_kernel<<<1, 32, 0, reinterpret_cast<cudaStream_t>(stream)>>>(limit, status);
    return from_cuda(cudaGetLastError());
}
