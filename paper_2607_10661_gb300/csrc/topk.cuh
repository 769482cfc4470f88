// Internal launcher of the per-node top-k kernel (not part of the C ABI).
#pragma once
#include <cuda_runtime.h>

#include <cstdint>

namespace ptd {
// Launched with programmatic stream serialization: the kernel waits for the stream's previous
// grid before its first global access and lets the next grid be placed early.
cudaError_t launch_topk(const void* logits, bool bf16, int64_t rows, int vocab, int64_t row_stride, int k,
                        int32_t* out_idx, float* out_val, int32_t* dev_status, cudaStream_t stream);
}  // namespace ptd
