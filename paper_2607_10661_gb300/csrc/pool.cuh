// Internal launchers of the candidate-pool kernels (not part of the C ABI).
#pragma once
#include <cuda_runtime.h>

#include <cstddef>
#include <cstdint>

namespace ptd {
constexpr int kPoolKids = 8;   // earliest children a pool node keeps for retrieval
size_t pool_bytes(int capacity);
cudaError_t pool_init(void* pool, int capacity, cudaStream_t stream);
cudaError_t launch_pool_merge(void* pool, int capacity, int max_load, int step, const int32_t* count,
                              const int32_t* parents, const int32_t* tokens, int32_t* dev_status, cudaStream_t stream);
cudaError_t launch_pool_retrieve(const void* pool, int capacity, const int32_t* root_token, int width, int max_depth,
                                 int max_nodes, int32_t* out_count, int32_t* out_parents, int32_t* out_tokens,
                                 cudaStream_t stream);
}  // namespace ptd
