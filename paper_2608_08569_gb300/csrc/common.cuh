// Internal helpers shared by the VoxZip kernels (not part of the C ABI).
#pragma once

#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "../../include/voxzip.h"

namespace voxzip {

constexpr int kMaxGroup = 16;  // largest GQA group (Hq / Hkv) the decode kernels take

// Element access for the two cache dtypes. Loads widen to fp32; stores round to nearest even.
template <typename T> struct Elem;

template <> struct Elem<float> {
    static __device__ __forceinline__ float to_f(float x) { return x; }
    static __device__ __forceinline__ float from_f(float x) { return x; }
};

template <> struct Elem<__nv_bfloat16> {
    static __device__ __forceinline__ float to_f(__nv_bfloat16 x) { return __bfloat162float(x); }
    static __device__ __forceinline__ __nv_bfloat16 from_f(float x) { return __float2bfloat16_rn(x); }
};

// Four consecutive elements as fp32 (D is a multiple of 4, rows 8- or 16-byte aligned).
__device__ __forceinline__ float4 load4(const float *p) { return *reinterpret_cast<const float4 *>(p); }
__device__ __forceinline__ float4 load4(const __nv_bfloat16 *p) {
    uint2 u = *reinterpret_cast<const uint2 *>(p);
    float4 r;
    r.x = __uint_as_float(u.x << 16);
    r.y = __uint_as_float(u.x & 0xffff0000u);
    r.z = __uint_as_float(u.y << 16);
    r.w = __uint_as_float(u.y & 0xffff0000u);
    return r;
}
__device__ __forceinline__ void store4(float *p, float4 v) { *reinterpret_cast<float4 *>(p) = v; }
__device__ __forceinline__ void store4(__nv_bfloat16 *p, float4 v) {
    __nv_bfloat162 a = __floats2bfloat162_rn(v.x, v.y);
    __nv_bfloat162 b = __floats2bfloat162_rn(v.z, v.w);
    uint2 u;
    u.x = *reinterpret_cast<uint32_t *>(&a);
    u.y = *reinterpret_cast<uint32_t *>(&b);
    *reinterpret_cast<uint2 *>(p) = u;
}

__device__ __forceinline__ void raise_status(int32_t *status, uint32_t bits) {
    atomicOr(reinterpret_cast<unsigned int *>(status), bits);
}

// Builds with -DVOXZIP_CHECKED range-check the indices of the accesses this guards: a violation
// sets VOXZIP_DEV_BOUNDS and the guarded access is skipped (never a trap). Regular builds compile
// the checks out.
#ifdef VOXZIP_CHECKED
#define VOXZIP_IN_RANGE(status, cond) ((cond) ? true : (voxzip::raise_status((status), VOXZIP_DEV_BOUNDS), false))
#else
#define VOXZIP_IN_RANGE(status, cond) true
#endif

// Unit index helpers. Units of a call are ordered (layer_local, b, h) to match the per-layer
// activation layout [layer][B][heads][D]; cache arrays are ordered (b, layer, h).
struct UnitIdx {
    int l_local, l, b, h;
    int64_t cache_unit;  // (b * L + l) * Hkv + h
};
__device__ __forceinline__ UnitIdx unit_of(int u, int B, int L, int Hkv, int layer_begin) {
    UnitIdx r;
    r.h = u % Hkv;
    r.b = (u / Hkv) % B;
    r.l_local = u / (Hkv * B);
    r.l = layer_begin + r.l_local;
    r.cache_unit = ((int64_t)r.b * L + r.l) * Hkv + r.h;
    return r;
}

}  // namespace voxzip

// Host-side launchers (one per kernel family), defined in their .cu files; status is the
// device status word's address on the current device.
namespace voxzip {
cudaError_t launch_anchor_fuse(const voxzip_cache_desc &d, const void *k_prefill, const void *v_prefill,
                               int32_t prefill_stride, const int32_t *in_len, const int32_t *audio_begin,
                               const int32_t *audio_len, const int32_t *span_off, int32_t num_spans,
                               const int32_t *span_start, const int32_t *span_end,
                               const int32_t *span_groups, const void *anchor_k, const void *anchor_v,
                               int32_t anchor_stride, void *k_cache, void *v_cache, float *score,
                               int32_t *pos, int32_t *len, int32_t *slot_map, void *workspace,
                               int32_t *status, cudaStream_t stream);
size_t anchor_fuse_workspace_bytes(const voxzip_cache_desc &d, int32_t prefill_stride, int32_t num_spans);

cudaError_t launch_decode(const voxzip_cache_desc &d, int32_t layer_begin, int32_t layer_count,
                          const void *q, const void *k_new, const void *v_new, const int32_t *new_pos,
                          void *k_cache, void *v_cache, float *score, int32_t *pos, int32_t *len,
                          float gamma, float sm_scale, int32_t max_len, void *out, int32_t *status,
                          cudaStream_t stream, bool *unsupported);

bool decode_mma_supported(const voxzip_cache_desc &d);
cudaError_t launch_decode_mma(const voxzip_cache_desc &d, int32_t layer_begin, int32_t layer_count, const void *q,
                              const void *k_new, const void *v_new, const int32_t *new_pos, void *k_cache,
                              void *v_cache, float *score, int32_t *pos, int32_t *len, float gamma, float sm_scale,
                              int32_t max_len, void *out, int32_t *status, cudaStream_t stream, bool *unsupported);

cudaError_t launch_evict(const voxzip_cache_desc &d, int32_t layer_begin, int32_t layer_count,
                         void *k_cache, void *v_cache, float *score, int32_t *pos, int32_t *len,
                         const int32_t *budget, int32_t sink, float recent_frac, int32_t *status,
                         cudaStream_t stream);
}  // namespace voxzip
