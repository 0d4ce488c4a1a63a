// Launcher of the eviction under a policy (evict.cu), called by the C ABI (api.cu).
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

#include "voxzip.h"

namespace voxzip {

// SMs of the current device (anchor_fuse.cu; looked up once per device).
int sm_count();

cudaError_t launch_evict_policy(const voxzip_cache_desc &d, int32_t layer_begin, int32_t layer_count,
                                void *k_cache, void *v_cache, float *score, int32_t *pos, int32_t *len,
                                const int32_t *budget, const voxzip_evict_policy &policy, int32_t *status,
                                cudaStream_t stream);

}  // namespace voxzip
