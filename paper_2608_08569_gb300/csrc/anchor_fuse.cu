// Stage 1 of VoxZip (Sec. 3.2.1): semantic-anchored fusion of the prefilled K/V cache.
//
// Three kernels, all launched on the caller's stream:
//   span_scan   one CTA per sequence: validates the semantic set (sorted, non-overlapping spans
//               inside the audio region) and scans, per span, the slot shift
//               delta = min(n_groups, l) - l and the anchor-row offset (prefix of n_groups);
//   slot_map    one thread per prefill token: the output slot of the token (Eq. 4 grouping with
//               group j = [floor(j*l/g), floor((j+1)*l/g)), Eq. 5 chronological order); the first
//               token of each slot records the slot's source range start and anchor row;
//   fuse_rows   one warp-slice per output slot of every (layer, kv-head) unit: the fp32 mean of
//               the slot's source rows (a copy when the range has one row) plus the anchor row,
//               rounded once to the cache dtype; K and V in the same pass; pos and score = 0.
// Output slots tile the prompt into contiguous ranges in order, so a slot is fully described by
// the first token of its range; the range ends where the next slot's begins.
#include "common.cuh"

namespace voxzip {
namespace {

constexpr int kScanThreads = 512;
constexpr int kMapThreads = 256;
constexpr int kFuseWarps = 8;
constexpr int kSlotsPerWarp = 8;

struct FuseWorkspace {
    int32_t *seq_len;        // [B] stage-1 length, -1 when the sequence is skipped
    int32_t *delta_prefix;   // [num_spans] exclusive prefix of (g - l) within the sequence
    int32_t *anchor_prefix;  // [num_spans] exclusive prefix of n_groups within the sequence
    int32_t *slot_src;       // [B][stride + 1] first prefill token of each slot, then in_len
    int32_t *slot_anchor;    // [B][stride] anchor row of each slot, -1 for copied rows
};

__host__ __device__ inline size_t align256(size_t x) { return (x + 255) & ~size_t(255); }

__host__ __device__ inline size_t carve(const voxzip_cache_desc &d, int32_t stride, int32_t num_spans,
                                        char *base, FuseWorkspace *ws) {
    size_t off = 0;
    auto take = [&](size_t bytes) {
        char *p = base + off;
        off += align256(bytes);
        return reinterpret_cast<int32_t *>(p);
    };
    int32_t *a = take(sizeof(int32_t) * (size_t)d.batch);
    int32_t *b = take(sizeof(int32_t) * (size_t)num_spans);
    int32_t *c = take(sizeof(int32_t) * (size_t)num_spans);
    int32_t *e = take(sizeof(int32_t) * (size_t)d.batch * ((size_t)stride + 1));
    int32_t *f = take(sizeof(int32_t) * (size_t)d.batch * (size_t)stride);
    if (ws) {
        ws->seq_len = a;
        ws->delta_prefix = b;
        ws->anchor_prefix = c;
        ws->slot_src = e;
        ws->slot_anchor = f;
    }
    return off;
}

// Block-wide exclusive scan of one int per thread; returns the block total in *total.
__device__ int block_excl_scan(int v, int *total) {
    __shared__ int warp_sums[32];
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nw = blockDim.x >> 5;
    int x = v;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        int y = __shfl_up_sync(0xffffffffu, x, o);
        if (lane >= o) x += y;
    }
    if (lane == 31) warp_sums[warp] = x;
    __syncthreads();
    if (warp == 0) {
        int s = lane < nw ? warp_sums[lane] : 0;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            int y = __shfl_up_sync(0xffffffffu, s, o);
            if (lane >= o) s += y;
        }
        warp_sums[lane] = s;  // inclusive over warps
    }
    __syncthreads();
    const int warp_off = warp > 0 ? warp_sums[warp - 1] : 0;
    *total = warp_sums[nw - 1];
    __syncthreads();
    return warp_off + x - v;
}

__global__ void __launch_bounds__(kScanThreads)
span_scan_kernel(int32_t B, int32_t stride, int32_t capacity, int32_t num_spans, int32_t anchor_stride,
                 bool has_anchor, const int32_t *__restrict__ in_len, const int32_t *__restrict__ audio_begin,
                 const int32_t *__restrict__ audio_len, const int32_t *__restrict__ span_off,
                 const int32_t *__restrict__ span_start, const int32_t *__restrict__ span_end,
                 const int32_t *__restrict__ span_groups, FuseWorkspace ws, int32_t *status) {
    const int b = blockIdx.x;
    __shared__ int bad;
    if (threadIdx.x == 0) bad = 0;
    __syncthreads();
    const int32_t n_in = in_len[b], ab = audio_begin[b], al = audio_len[b];
    const int32_t s0 = span_off[b], s1 = span_off[b + 1];
    const bool header_ok = n_in >= 0 && n_in <= stride && ab >= 0 && al >= 0 &&
                           (int64_t)ab + al <= n_in && s0 >= 0 && s0 <= s1 && s1 <= num_spans;
    if (!header_ok) {
        if (threadIdx.x == 0) {
            ws.seq_len[b] = -1;
            raise_status(status, VOXZIP_DEV_BAD_SPANS);
        }
        return;
    }
    int carry_delta = 0, carry_groups = 0;
    for (int base = s0; base < s1; base += blockDim.x) {
        const int i = base + threadIdx.x;
        int delta = 0, groups = 0;
        if (i < s1) {
            const int32_t st = span_start[i], en = span_end[i], ng = span_groups[i];
            const int32_t prev_end = i > s0 ? span_end[i - 1] : ab;
            if (st < prev_end || en < st || en > ab + al || ng < 1) bad = 1;
            const int32_t l = en - st;
            delta = (ng < l ? ng : l) - l;
            groups = ng;
        }
        int tot_d, tot_g;
        const int ex_d = block_excl_scan(delta, &tot_d);
        const int ex_g = block_excl_scan(groups, &tot_g);
        if (i < s1) {
            ws.delta_prefix[i] = carry_delta + ex_d;
            ws.anchor_prefix[i] = carry_groups + ex_g;
        }
        carry_delta += tot_d;
        carry_groups += tot_g;
    }
    __syncthreads();
    if (threadIdx.x == 0) {
        const int64_t out_len = (int64_t)n_in + carry_delta;
        if (bad || (has_anchor && carry_groups > anchor_stride)) {
            ws.seq_len[b] = -1;
            raise_status(status, VOXZIP_DEV_BAD_SPANS);
        } else if (out_len > capacity) {
            ws.seq_len[b] = -1;
            raise_status(status, VOXZIP_DEV_CAPACITY);
        } else {
            ws.seq_len[b] = (int32_t)out_len;
        }
    }
}

__global__ void __launch_bounds__(kMapThreads)
slot_map_kernel(int32_t stride, const int32_t *__restrict__ in_len, const int32_t *__restrict__ span_off,
                const int32_t *__restrict__ span_start, const int32_t *__restrict__ span_end,
                const int32_t *__restrict__ span_groups, FuseWorkspace ws, int32_t *__restrict__ slot_map) {
    const int b = blockIdx.y;
    const int32_t t = blockIdx.x * blockDim.x + threadIdx.x;
    const int32_t out_len = ws.seq_len[b];
    const int32_t n_in = in_len[b];
    if (out_len < 0 || t >= n_in) return;
    const int32_t s0 = span_off[b], s1 = span_off[b + 1];
    // Last span with start <= t.
    int lo = s0, hi = s1;  // answer in [s0 - 1, s1)
    while (lo < hi) {
        const int mid = (lo + hi) >> 1;
        if (span_start[mid] <= t) lo = mid + 1;
        else hi = mid;
    }
    const int i = lo - 1;
    int32_t slot, anchor = -1;
    bool first;
    if (i >= s0 && t < span_end[i]) {
        const int64_t st = span_start[i], l = span_end[i] - st;
        const int64_t ng = span_groups[i];
        const int64_t g = ng < l ? ng : l;
        const int64_t r = t - st;
        const int64_t j = ((r + 1) * g - 1) / l;  // group j holds r iff floor(j*l/g) <= r < floor((j+1)*l/g)
        slot = (int32_t)(st + ws.delta_prefix[i] + j);
        first = r == (j * l) / g;
        anchor = (int32_t)(ws.anchor_prefix[i] + j);
    } else {
        const int32_t shift = i >= s0 ? ws.delta_prefix[i] + (min(span_groups[i], span_end[i] - span_start[i]) -
                                                             (span_end[i] - span_start[i]))
                                      : 0;
        slot = t + shift;
        first = true;
    }
    if (slot_map) slot_map[(int64_t)b * stride + t] = slot;
    if (first) {
        ws.slot_src[(int64_t)b * (stride + 1) + slot] = t;
        ws.slot_anchor[(int64_t)b * stride + slot] = anchor;
    }
    if (t == n_in - 1) ws.slot_src[(int64_t)b * (stride + 1) + out_len] = n_in;
}

template <typename T, int D>
__global__ void __launch_bounds__(kFuseWarps * 32)
fuse_rows_kernel(int32_t B, int32_t L, int32_t Hkv, int32_t C, int32_t stride, int32_t anchor_stride,
                 const T *__restrict__ k_prefill, const T *__restrict__ v_prefill,
                 const T *__restrict__ anchor_k, const T *__restrict__ anchor_v, FuseWorkspace ws,
                 T *__restrict__ k_cache, T *__restrict__ v_cache, float *__restrict__ score,
                 int32_t *__restrict__ pos, int32_t *__restrict__ len) {
    constexpr int kLanesPerRow = D / 4;          // each lane owns 4 consecutive elements
    constexpr int kRowsPerWarp = 32 / kLanesPerRow;
    const int u = blockIdx.y;                    // cache unit (b, l, h)
    const int b = u / (L * Hkv);
    const int32_t out_len = ws.seq_len[b];
    if (blockIdx.x == 0 && threadIdx.x == 0) len[u] = out_len < 0 ? 0 : out_len;
    if (out_len < 0) return;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int sub = lane / kLanesPerRow, e = (lane % kLanesPerRow) * 4;
    const int64_t in_base = (int64_t)u * stride * D;
    const int64_t out_base = (int64_t)u * C * D;
    const int64_t anc_base = (int64_t)u * anchor_stride * D;
    const int32_t *src = ws.slot_src + (int64_t)b * (stride + 1);
    const int32_t *anc = ws.slot_anchor + (int64_t)b * stride;
    const int slot0 = (blockIdx.x * kFuseWarps + warp) * kSlotsPerWarp * kRowsPerWarp;
    for (int k = 0; k < kSlotsPerWarp; ++k) {
        const int s = slot0 + k * kRowsPerWarp + sub;
        if (s >= out_len) break;
        const int32_t r0 = src[s], r1 = src[s + 1];
        float4 sk = make_float4(0.f, 0.f, 0.f, 0.f), sv = sk;
        for (int32_t r = r0; r < r1; ++r) {
            const float4 a = load4(k_prefill + in_base + (int64_t)r * D + e);
            const float4 c = load4(v_prefill + in_base + (int64_t)r * D + e);
            sk.x += a.x; sk.y += a.y; sk.z += a.z; sk.w += a.w;
            sv.x += c.x; sv.y += c.y; sv.z += c.z; sv.w += c.w;
        }
        if (r1 - r0 > 1) {
            const float cnt = (float)(r1 - r0);
            sk.x = __fdiv_rn(sk.x, cnt); sk.y = __fdiv_rn(sk.y, cnt);
            sk.z = __fdiv_rn(sk.z, cnt); sk.w = __fdiv_rn(sk.w, cnt);
            sv.x = __fdiv_rn(sv.x, cnt); sv.y = __fdiv_rn(sv.y, cnt);
            sv.z = __fdiv_rn(sv.z, cnt); sv.w = __fdiv_rn(sv.w, cnt);
        }
        const int32_t a_row = anc[s];
        if (anchor_k != nullptr && a_row >= 0) {
            const float4 ak = load4(anchor_k + anc_base + (int64_t)a_row * D + e);
            const float4 av = load4(anchor_v + anc_base + (int64_t)a_row * D + e);
            sk.x = __fadd_rn(sk.x, ak.x); sk.y = __fadd_rn(sk.y, ak.y);
            sk.z = __fadd_rn(sk.z, ak.z); sk.w = __fadd_rn(sk.w, ak.w);
            sv.x = __fadd_rn(sv.x, av.x); sv.y = __fadd_rn(sv.y, av.y);
            sv.z = __fadd_rn(sv.z, av.z); sv.w = __fadd_rn(sv.w, av.w);
        }
        store4(k_cache + out_base + (int64_t)s * D + e, sk);
        store4(v_cache + out_base + (int64_t)s * D + e, sv);
        if (e == 0) {
            pos[(int64_t)u * C + s] = r0;
            score[(int64_t)u * C + s] = 0.f;
        }
    }
}

template <typename T, int D>
cudaError_t launch_fuse_rows(const voxzip_cache_desc &d, int32_t stride, int32_t anchor_stride,
                             const void *kp, const void *vp, const void *ak, const void *av,
                             const FuseWorkspace &ws, void *kc, void *vc, float *score, int32_t *pos,
                             int32_t *len, cudaStream_t stream) {
    constexpr int kRowsPerWarp = 32 / (D / 4);
    const int slots_per_block = kFuseWarps * kSlotsPerWarp * kRowsPerWarp;
    const int64_t units = (int64_t)d.batch * d.layers * d.kv_heads;
    dim3 grid((unsigned)((stride + slots_per_block - 1) / slots_per_block), (unsigned)units);
    if (grid.x == 0) grid.x = 1;
    fuse_rows_kernel<T, D><<<grid, kFuseWarps * 32, 0, stream>>>(
        d.batch, d.layers, d.kv_heads, d.capacity, stride, anchor_stride, (const T *)kp, (const T *)vp,
        (const T *)ak, (const T *)av, ws, (T *)kc, (T *)vc, score, pos, len);
    return cudaGetLastError();
}

}  // namespace

size_t anchor_fuse_workspace_bytes(const voxzip_cache_desc &d, int32_t prefill_stride, int32_t num_spans) {
    return carve(d, prefill_stride, num_spans, nullptr, nullptr);
}

cudaError_t launch_anchor_fuse(const voxzip_cache_desc &d, const void *k_prefill, const void *v_prefill,
                               int32_t prefill_stride, const int32_t *in_len, const int32_t *audio_begin,
                               const int32_t *audio_len, const int32_t *span_off, int32_t num_spans,
                               const int32_t *span_start, const int32_t *span_end,
                               const int32_t *span_groups, const void *anchor_k, const void *anchor_v,
                               int32_t anchor_stride, void *k_cache, void *v_cache, float *score,
                               int32_t *pos, int32_t *len, int32_t *slot_map, void *workspace,
                               int32_t *status, cudaStream_t stream) {
    FuseWorkspace ws;
    carve(d, prefill_stride, num_spans, static_cast<char *>(workspace), &ws);
    const bool has_anchor = anchor_k != nullptr;
    span_scan_kernel<<<d.batch, kScanThreads, 0, stream>>>(
        d.batch, prefill_stride, d.capacity, num_spans, anchor_stride, has_anchor, in_len, audio_begin,
        audio_len, span_off, span_start, span_end, span_groups, ws, status);
    cudaError_t err = cudaGetLastError();
    if (err != cudaSuccess) return err;
    dim3 grid_map((unsigned)((prefill_stride + kMapThreads - 1) / kMapThreads), (unsigned)d.batch);
    slot_map_kernel<<<grid_map, kMapThreads, 0, stream>>>(prefill_stride, in_len, span_off, span_start,
                                                          span_end, span_groups, ws, slot_map);
    err = cudaGetLastError();
    if (err != cudaSuccess) return err;
    const bool bf16 = d.dtype == VOXZIP_BF16;
    if (d.head_dim == 128)
        return bf16 ? launch_fuse_rows<__nv_bfloat16, 128>(d, prefill_stride, anchor_stride, k_prefill, v_prefill,
                                                            anchor_k, anchor_v, ws, k_cache, v_cache, score, pos,
                                                            len, stream)
                    : launch_fuse_rows<float, 128>(d, prefill_stride, anchor_stride, k_prefill, v_prefill,
                                                   anchor_k, anchor_v, ws, k_cache, v_cache, score, pos, len,
                                                   stream);
    return bf16 ? launch_fuse_rows<__nv_bfloat16, 64>(d, prefill_stride, anchor_stride, k_prefill, v_prefill,
                                                       anchor_k, anchor_v, ws, k_cache, v_cache, score, pos, len,
                                                       stream)
                : launch_fuse_rows<float, 64>(d, prefill_stride, anchor_stride, k_prefill, v_prefill, anchor_k,
                                              anchor_v, ws, k_cache, v_cache, score, pos, len, stream);
}

}  // namespace voxzip
