// Internal launcher of the sampling-verification kernel (not part of the C ABI).
#pragma once
#include <cuda_runtime.h>

#include <cstdint>

namespace ptd {
cudaError_t launch_verify_sampling(const int32_t* node_offsets, const int32_t* parents, const int32_t* tokens,
                                   const void* logits, bool bf16, int vocab, int64_t row_stride, float inv_temp,
                                   const float* u_accept, const float* u_bonus, int batch, int n_total, int max_nodes,
                                   int32_t* accepted, int32_t* accept_len, int32_t* bonus, int32_t* dev_status,
                                   cudaStream_t stream);
}  // namespace ptd
