// Stage-2 decode step of VoxZip: cache append (Eq. 1), GQA attention (Eq. 2) and the temporally
// decayed accumulated score (Eq. 6), fused so that every cached K and V row is read once.
//
// One thread-block cluster of S CTAs per (layer, sequence, kv-head) unit; CTA r of the cluster
// owns the contiguous token range [r*ceil(n/S), (r+1)*ceil(n/S)). Per CTA:
//   1. the CTA owning slot n (the new token) appends k_new, v_new and its position;
//   2. logits of the G query heads for its tokens go to shared memory (log2 domain);
//   3. per-head maxima are exchanged through distributed shared memory (cluster barrier);
//   4. p = 2^(logit - max) in place, local sums, and the partial P V for its tokens;
//   5. per-head sums are exchanged; the CTA rewrites the scores of its tokens as
//      gamma * s + sum_h p_h / Z_h and combines one slice of the G x D outputs from all CTAs.
// The score update needs the global softmax normaliser before any score is written; keeping
// the logits of a CTA's range in shared memory between the two exchanges is what lets K be read
// once per step.
#include <cooperative_groups.h>

#include "common.cuh"

namespace cg = cooperative_groups;

namespace voxzip {
namespace {

constexpr int kThreads = 256;
constexpr int kWarps = kThreads / 32;
constexpr int kTargetTokensPerCta = 256;
constexpr int kMaxCluster = 16;
constexpr size_t kMaxSmem = 227 * 1024;

struct DecodeParams {
    const void *q, *k_new, *v_new;
    const int32_t *new_pos;
    void *k_cache, *v_cache;
    float *score;
    int32_t *pos, *len;
    void *out;
    int32_t *status;
    int32_t B, L, Hq, Hkv, G, C, layer_begin, chunk_cap;
    float gamma, scale_log2;
};

__device__ __forceinline__ float warp_max(float v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
    return v;
}
__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    return v;
}

template <typename T, int D>
__global__ void __launch_bounds__(kThreads) decode_kernel(const DecodeParams p) {
    constexpr int kLanesPerRow = D / 4;           // lanes covering one row, 4 elements each
    constexpr int kRowsPerWarp = 32 / kLanesPerRow;
    constexpr int kHeadsPerPass = kThreads / kLanesPerRow;

    cg::cluster_group cluster = cg::this_cluster();
    const int S = (int)cluster.num_blocks();
    const int rank = (int)cluster.block_rank();
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int G = p.G, D_ = D;

    extern __shared__ float smem[];
    float *qs = smem;                                   // [G][D], pre-scaled by scale*log2(e)
    float *os = qs + G * D_;                            // [G][D] partial outputs
    float *stat = os + G * D_;                          // mx[16] zs[16] mg[16] rz[16]
    float *mx = stat, *zs = stat + 16, *mg = stat + 32, *rz = stat + 48;
    float *lg = stat + 64;                              // [G][chunk_cap] logits, then p

    const UnitIdx ui = unit_of(blockIdx.y, p.B, p.L, p.Hkv, p.layer_begin);
    const int32_t n_old = p.len[ui.cache_unit];
    const int32_t n = n_old + 1;
    if (n_old < 0 || n > p.C) {  // same decision in every CTA of the cluster
        if (rank == 0 && tid == 0) raise_status(p.status, VOXZIP_DEV_CAPACITY);
        return;
    }
    const int chunk = (n + S - 1) / S;
    if (chunk > p.chunk_cap) {
        if (rank == 0 && tid == 0) raise_status(p.status, VOXZIP_DEV_LEN_HINT);
        return;
    }
    const int j0 = min(n, rank * chunk), j1 = min(n, j0 + chunk), cnt = j1 - j0;

    const int64_t act_row = (int64_t)ui.l_local * p.B + ui.b;   // [layer_local][B] activation row
    const T *qg = static_cast<const T *>(p.q) + (act_row * p.Hq + (int64_t)ui.h * G) * D;
    T *kc = static_cast<T *>(p.k_cache) + ui.cache_unit * p.C * D;
    T *vc = static_cast<T *>(p.v_cache) + ui.cache_unit * p.C * D;
    float *sc = p.score + ui.cache_unit * p.C;

    for (int i = tid; i < G * D; i += kThreads) qs[i] = Elem<T>::to_f(qg[i]) * p.scale_log2;
    // Eq. 1: the CTA that owns slot n-1 appends the new token.
    if (j0 <= n - 1 && n - 1 < j1) {
        const T *kn = static_cast<const T *>(p.k_new) + (act_row * p.Hkv + ui.h) * D;
        const T *vn = static_cast<const T *>(p.v_new) + (act_row * p.Hkv + ui.h) * D;
        for (int i = tid; i < D; i += kThreads) {
            kc[(int64_t)(n - 1) * D + i] = kn[i];
            vc[(int64_t)(n - 1) * D + i] = vn[i];
        }
        if (tid == 0) p.pos[ui.cache_unit * p.C + n - 1] = p.new_pos[ui.b];
    }
    __syncthreads();

    // Logits for this CTA's tokens (Eq. 2 numerator), log2 domain.
    const int sub = lane / kLanesPerRow, e = (lane % kLanesPerRow) * 4;
    for (int base = warp * kRowsPerWarp; base < cnt; base += kWarps * kRowsPerWarp) {
        const int jj = base + sub;
        const bool valid = jj < cnt;
        const float4 k4 = valid ? load4(kc + (int64_t)(j0 + jj) * D + e) : make_float4(0.f, 0.f, 0.f, 0.f);
        float acc[kMaxGroup];
#pragma unroll
        for (int g = 0; g < kMaxGroup; ++g) {
            if (g < G) {
                const float *qr = qs + g * D + e;
                acc[g] = qr[0] * k4.x + qr[1] * k4.y + qr[2] * k4.z + qr[3] * k4.w;
            }
        }
#pragma unroll
        for (int g = 0; g < kMaxGroup; ++g) {
            if (g < G) {
#pragma unroll
                for (int o = kLanesPerRow / 2; o > 0; o >>= 1) acc[g] += __shfl_xor_sync(0xffffffffu, acc[g], o);
            }
        }
        if (valid && (lane % kLanesPerRow) == 0) {
#pragma unroll
            for (int g = 0; g < kMaxGroup; ++g)
                if (g < G) lg[g * p.chunk_cap + jj] = acc[g];
        }
    }
    __syncthreads();

    for (int g = warp; g < G; g += kWarps) {
        float m = -INFINITY;
        for (int i = lane; i < cnt; i += 32) m = fmaxf(m, lg[g * p.chunk_cap + i]);
        m = warp_max(m);
        if (lane == 0) mx[g] = m;
    }
    cluster.sync();
    if (tid < G) {
        float m = -INFINITY;
        for (int r = 0; r < S; ++r) m = fmaxf(m, *cluster.map_shared_rank(&mx[tid], r));
        mg[tid] = m;
    }
    __syncthreads();

    for (int g = 0; g < G; ++g)
        for (int i = tid; i < cnt; i += kThreads) lg[g * p.chunk_cap + i] = exp2f(lg[g * p.chunk_cap + i] - mg[g]);
    __syncthreads();
    for (int g = warp; g < G; g += kWarps) {
        float z = 0.f;
        for (int i = lane; i < cnt; i += 32) z += lg[g * p.chunk_cap + i];
        z = warp_sum(z);
        if (lane == 0) zs[g] = z;
    }
    // Partial P V over this CTA's tokens.
    {
        const int ed = (tid % kLanesPerRow) * 4;
        for (int g = tid / kLanesPerRow; g < G; g += kHeadsPerPass) {
            float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
            const float *pr = lg + g * p.chunk_cap;
            for (int j = 0; j < cnt; ++j) {
                const float pj = pr[j];
                const float4 v = load4(vc + (int64_t)(j0 + j) * D + ed);
                acc.x += pj * v.x; acc.y += pj * v.y; acc.z += pj * v.z; acc.w += pj * v.w;
            }
            float *o = os + g * D + ed;
            o[0] = acc.x; o[1] = acc.y; o[2] = acc.z; o[3] = acc.w;
        }
    }
    cluster.sync();
    if (tid < G) {
        float z = 0.f;
        for (int r = 0; r < S; ++r) z += *cluster.map_shared_rank(&zs[tid], r);
        rz[tid] = 1.f / z;
    }
    __syncthreads();

    // Eq. 6: A = gamma * [A, 0] + sum over the group's heads of the softmax.
    for (int i = tid; i < cnt; i += kThreads) {
        const int j = j0 + i;
        const float prev = (j == n - 1) ? 0.f : sc[j];
        float add = 0.f;
        for (int g = 0; g < G; ++g) add += lg[g * p.chunk_cap + i] * rz[g];
        sc[j] = p.gamma * prev + add;
    }
    // Combine the partial outputs of all CTAs; CTA r writes slice r of the G*D outputs.
    {
        const int total = G * D, per = (total + S - 1) / S;
        const int lo = rank * per, hi = min(total, lo + per);
        T *og = static_cast<T *>(p.out) + (act_row * p.Hq + (int64_t)ui.h * G) * D;
        for (int i = lo + tid; i < hi; i += kThreads) {
            float o = 0.f;
            for (int r = 0; r < S; ++r) o += *cluster.map_shared_rank(&os[i], r);
            og[i] = Elem<T>::from_f(o * rz[i / D]);
        }
    }
    cluster.sync();  // no CTA leaves while others may still read its shared memory
    if (rank == 0 && tid == 0) p.len[ui.cache_unit] = n;
}

template <typename T, int D>
cudaError_t launch_t(const DecodeParams &prm, int S, size_t smem, int units, cudaStream_t stream) {
    auto kern = decode_kernel<T, D>;
    static bool configured = false;  // attributes are per function; set once per process
    if (!configured) {
        cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kMaxSmem);
        if (e != cudaSuccess) return e;
        e = cudaFuncSetAttribute(kern, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
        if (e != cudaSuccess) return e;
        configured = true;
    }
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)S, (unsigned)units, 1);
    cfg.blockDim = dim3(kThreads, 1, 1);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = stream;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = (unsigned)S;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, kern, prm);
}

}  // namespace

cudaError_t launch_decode(const voxzip_cache_desc &d, int32_t layer_begin, int32_t layer_count,
                          const void *q, const void *k_new, const void *v_new, const int32_t *new_pos,
                          void *k_cache, void *v_cache, float *score, int32_t *pos, int32_t *len,
                          float gamma, float sm_scale, int32_t max_len, void *out, int32_t *status,
                          cudaStream_t stream, bool *unsupported) {
    *unsupported = false;
    if (decode_mma_supported(d)) {
        cudaError_t e = launch_decode_mma(d, layer_begin, layer_count, q, k_new, v_new, new_pos, k_cache, v_cache,
                                          score, pos, len, gamma, sm_scale, max_len, out, status, stream,
                                          unsupported);
        if (!*unsupported) return e;
        *unsupported = false;  // shape outside the tensor-core kernel's limits: the generic kernel runs
    }
    const int G = d.q_heads / d.kv_heads;
    const int units = layer_count * d.batch * d.kv_heads;
    const int nmax = (max_len > 0 && max_len < d.capacity) ? max_len : d.capacity;
    int S = 1;
    while (S < kMaxCluster && (nmax + S - 1) / S > kTargetTokensPerCta) S <<= 1;
    auto smem_for = [&](int s) {
        const int cap = (nmax + s - 1) / s;
        return sizeof(float) * ((size_t)2 * G * d.head_dim + 64 + (size_t)G * cap);
    };
    while (smem_for(S) > kMaxSmem && S < kMaxCluster) S <<= 1;
    if (smem_for(S) > kMaxSmem) {
        *unsupported = true;
        return cudaSuccess;
    }
    DecodeParams prm;
    prm.q = q; prm.k_new = k_new; prm.v_new = v_new; prm.new_pos = new_pos;
    prm.k_cache = k_cache; prm.v_cache = v_cache; prm.score = score; prm.pos = pos; prm.len = len;
    prm.out = out; prm.status = status;
    prm.B = d.batch; prm.L = d.layers; prm.Hq = d.q_heads; prm.Hkv = d.kv_heads; prm.G = G;
    prm.C = d.capacity; prm.layer_begin = layer_begin; prm.chunk_cap = (nmax + S - 1) / S;
    prm.gamma = gamma;
    const float scale = sm_scale > 0.f ? sm_scale : 1.0f / sqrtf((float)d.head_dim);
    prm.scale_log2 = scale * 1.4426950408889634f;  // log2(e): exp(x) = 2^(x log2 e)
    const size_t smem = smem_for(S);
    const bool bf16 = d.dtype == VOXZIP_BF16;
    if (d.head_dim == 128)
        return bf16 ? launch_t<__nv_bfloat16, 128>(prm, S, smem, units, stream)
                    : launch_t<float, 128>(prm, S, smem, units, stream);
    return bf16 ? launch_t<__nv_bfloat16, 64>(prm, S, smem, units, stream)
                : launch_t<float, 64>(prm, S, smem, units, stream);
}

}  // namespace voxzip
