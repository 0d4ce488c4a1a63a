// Stage-1 fusion for callers that cannot allocate device memory.
//
// voxzip_anchor_fuse needs a caller-provided scratch workspace. Some callers cannot provide one:
// a host runtime whose device memory is entirely owned by another framework's pool, or an audio
// front-end that must not allocate once it is serving. This file gives them an entry point that
// allocates nothing: its scratch is a fixed array compiled into the library, which every GPU that
// loads the library holds until the process exits.
//
// Host code cannot pass the array's name to a kernel (on the host that name is only a stand-in,
// not a device address), so the device address is looked up once per device with
// cudaGetSymbolAddress, with that device current, on the first call made on it.
#include <atomic>

#include "common.cuh"

namespace {

constexpr size_t kScratchBytes = size_t(4) << 20;  // 4 MiB, shared by every call on a device

// The scratch itself. No entry needs to start at zero: every word a call reads was written earlier
// in the same call. Calls that overlap on the GPU (different streams, no ordering) share it and race.
static __device__ __align__(256) unsigned char g_fuse_scratch[kScratchBytes];

// The status word lives in api.cu; kernels of this file report through the same word.
constexpr int kMaxDevices = 64;
// Device address of g_fuse_scratch, per device. Two host threads making their first call on one
// device at once both look it up and store the same value; the atomic makes that well defined.
std::atomic<void *> g_scratch_addr[kMaxDevices];

voxzip_status scratch_address(void **out) {
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return VOXZIP_ECUDA;
    void *a = g_scratch_addr[dev].load(std::memory_order_acquire);
    if (a == nullptr) {
        if (cudaGetSymbolAddress(&a, g_fuse_scratch) != cudaSuccess || a == nullptr) return VOXZIP_ECUDA;
        g_scratch_addr[dev].store(a, std::memory_order_release);
    }
    *out = a;
    return VOXZIP_OK;
}

bool aligned16(const void *p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

}  // namespace

// Defined in api.cu: the status word's device address on the current device.
voxzip_status voxzip_status_word_address(int32_t **addr);

extern "C" voxzip_status voxzip_anchor_fuse_noalloc(
    const voxzip_cache_desc *desc, const void *k_prefill, const void *v_prefill, int32_t prefill_stride,
    const int32_t *in_len, const int32_t *audio_begin, const int32_t *audio_len, const int32_t *span_off,
    int32_t num_spans, const int32_t *span_start, const int32_t *span_end, const int32_t *span_groups,
    const void *anchor_k, const void *anchor_v, int32_t anchor_stride, void *k_cache, void *v_cache, float *score,
    int32_t *pos, int32_t *len, int32_t *slot_map, voxzip_stream_t stream) {
    // The same argument checks as voxzip_anchor_fuse, minus the workspace.
    if (desc == nullptr || desc->batch < 1 || desc->layers < 1 || desc->q_heads < 1 || desc->kv_heads < 1 ||
        desc->capacity < 1 || desc->q_heads % desc->kv_heads != 0 || (desc->head_dim != 64 && desc->head_dim != 128) ||
        (desc->dtype != VOXZIP_F32 && desc->dtype != VOXZIP_BF16))
        return VOXZIP_EINVAL;
    if (prefill_stride < 1 || num_spans < 0) return VOXZIP_EINVAL;
    if (!k_prefill || !v_prefill || !in_len || !audio_begin || !audio_len || !span_off || !k_cache || !v_cache ||
        !score || !pos || !len)
        return VOXZIP_EINVAL;
    if (num_spans > 0 && (!span_start || !span_end || !span_groups)) return VOXZIP_EINVAL;
    if ((anchor_k == nullptr) != (anchor_v == nullptr)) return VOXZIP_EINVAL;
    if (anchor_k && anchor_stride < 1) return VOXZIP_EINVAL;
    if (!aligned16(k_prefill) || !aligned16(v_prefill) || !aligned16(k_cache) || !aligned16(v_cache) ||
        (anchor_k && (!aligned16(anchor_k) || !aligned16(anchor_v))))
        return VOXZIP_EINVAL;
    if ((int64_t)desc->batch * desc->layers * desc->kv_heads > 65535) return VOXZIP_EUNSUPPORTED;
    // The one limit this entry point adds: the request's scratch must fit the fixed array.
    if (voxzip::anchor_fuse_workspace_bytes(*desc, prefill_stride, num_spans) > kScratchBytes) return VOXZIP_ESCRATCH;

    void *scratch = nullptr;
    voxzip_status st = scratch_address(&scratch);
    if (st != VOXZIP_OK) return st;
    int32_t *status = nullptr;
    st = voxzip_status_word_address(&status);
    if (st != VOXZIP_OK) return st;
    const cudaError_t e = voxzip::launch_anchor_fuse(
        *desc, k_prefill, v_prefill, prefill_stride, in_len, audio_begin, audio_len, span_off, num_spans, span_start,
        span_end, span_groups, anchor_k, anchor_v, anchor_stride, k_cache, v_cache, score, pos, len, slot_map, scratch,
        status, reinterpret_cast<cudaStream_t>(stream));
    return e == cudaSuccess ? VOXZIP_OK : VOXZIP_ECUDA;
}
