// Internal launcher of the per-node top-k kernel (not part of the C ABI).
#pragma once
#include <cuda_runtime.h>

#include <cstdint>

namespace ptd {
// early: the logits were complete before the stream's previous grid began (they are an input
// of the step whose attention launch precedes this one), so the kernel reads them without
// waiting for that grid; it still completes only after that grid has.  Any other caller
// passes false: the kernel then waits for the previous grid before its first global access.
cudaError_t launch_topk(const void* logits, bool bf16, int64_t rows, int vocab, int64_t row_stride, int k,
                        int32_t* out_idx, float* out_val, int32_t* dev_status, bool early, cudaStream_t stream);
}  // namespace ptd
