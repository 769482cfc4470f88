// Internal launcher of the LM-head + top-k kernel (not part of the C ABI).
#pragma once
#include <cuda.h>
#include <cuda_runtime.h>

#include <cstddef>
#include <cstdint>

namespace ptd {
constexpr int kLmMaxK = 16;
size_t lm_head_workspace_bytes(int ctas, int rows);
int lm_head_ctas(int num_sms, int vocab);
cudaError_t launch_lm_head_topk(const CUtensorMap& map_h, const CUtensorMap& map_w, int rows, int d_model, int vocab,
                                int k, int32_t* out_idx, float* out_val, void* workspace, int ctas,
                                int32_t* dev_status, cudaStream_t stream);
}  // namespace ptd
