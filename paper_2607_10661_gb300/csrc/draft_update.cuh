// Internal launcher of the draft-tree update kernel (not part of the C ABI).
#pragma once
#include <cuda_runtime.h>

#include <cstdint>

namespace ptd {
constexpr int kMaxExpand = 16;   // draft tokens a node may append per step
cudaError_t launch_draft_update(int batch, int in_stride, const int32_t* in_count, const int32_t* in_parents,
                                const int32_t* in_tokens, const int32_t* drafts, int draft_stride, int expand,
                                int width, int max_depth, int capacity, int32_t* out_count, int32_t* out_parents,
                                int32_t* out_tokens, int32_t* out_depths, int32_t* old_to_new, int32_t* dev_status,
                                cudaStream_t stream);
}  // namespace ptd
