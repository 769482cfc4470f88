// Internal launcher of the per-node top-k kernel (not part of the C ABI).
#pragma once
#include <cuda_runtime.h>

#include <cstdint>

namespace ptd {
// Greedy verification of each tree by the top-k cluster that completes the tree's rows (the
// step's tail): rows are the trees' nodes, back to back.
struct VerifyArgs {
  const int32_t* node_offsets;   // [batch + 1]
  const int32_t* parents;        // [n_total]
  const int32_t* tokens;         // [n_total]
  const int32_t* ctx_lens;       // [batch]
  unsigned int* counters;        // [batch] rows done per tree, zero before the launch
  int batch, n_total, max_nodes;
  int32_t* accepted;             // [batch][max_nodes]
  int32_t* accept_len;           // [batch]
  int32_t* bonus;                // [batch]
  int32_t* dev_status;
};

// Whether launch_topk can verify for these logits (bf16 rows within the clustered fast path).
bool topk_can_verify(bool bf16, int vocab);

// Launched with programmatic stream serialization: the kernel waits for the stream's previous
// grid before its first global access and lets the next grid be placed early.  With `va`
// (bf16 fast path only) it also verifies every tree, as ptd_verify_greedy on its column 0 would;
// the node_offsets / parents / tokens it reads must have been complete before the stream's
// previous grid began.
cudaError_t launch_topk(const void* logits, bool bf16, int64_t rows, int vocab, int64_t row_stride, int k,
                        int32_t* out_idx, float* out_val, int32_t* dev_status, const VerifyArgs* va,
                        cudaStream_t stream);
}  // namespace ptd
