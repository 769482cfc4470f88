// Internal launchers of the verification and compaction kernels (not part of the C ABI).
#pragma once
#include <cuda_runtime.h>

#include <cstdint>

namespace ptd {
cudaError_t launch_verify(const int32_t* node_offsets, const int32_t* parents, const int32_t* tokens,
                          const int32_t* target, int target_stride, int batch, int n_total, int max_nodes,
                          int32_t* accepted, int32_t* accept_len, int32_t* bonus, int32_t* dev_status,
                          cudaStream_t stream);
cudaError_t launch_compact(void* k, void* v, int row_bytes, int layers, int batch, int page_size, int seq_capacity,
                           int num_pages, const int32_t* block_table, int max_pages, const int32_t* ctx_lens,
                           const int32_t* accepted, const int32_t* accept_len, int max_nodes, int32_t* new_ctx,
                           cudaStream_t stream);
// Verification followed by compaction in one launch (the whole-step path).
cudaError_t launch_verify_compact(const int32_t* node_offsets, const int32_t* parents, const int32_t* tokens,
                                  const int32_t* target, int target_stride, int n_total, int max_nodes,
                                  int32_t* accepted, int32_t* accept_len, int32_t* bonus, int32_t* dev_status, void* k,
                                  void* v, int row_bytes, int layers, int batch, int page_size, int seq_capacity,
                                  int num_pages, const int32_t* block_table, int max_pages, const int32_t* ctx_lens,
                                  int32_t* new_ctx, cudaStream_t stream);
}  // namespace ptd
