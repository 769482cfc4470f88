// Internal launcher of the tree-position / rotary-encoding / K-V append kernel.
#pragma once
#include <cuda_runtime.h>

#include <cstdint>

namespace ptd {
constexpr int kMaxRopeHalf = 128;   // D / 2 for D <= 256
struct RopeFreqs {
  float hi[kMaxRopeHalf];           // base^(-2i/D) = hi + lo, from double
  float lo[kMaxRopeHalf];
};
cudaError_t launch_tree_rope(const int32_t* node_offsets, const int32_t* parents, const int32_t* ctx_lens,
                             int batch, int n_total, bool bf16, int head_dim, int hq, int hkv, void* q, const void* k,
                             const void* v, void* k_cache, void* v_cache, int layer_begin, int num_layers,
                             int page_size, int seq_capacity,
                             int num_pages, const int32_t* block_table, int max_pages, const RopeFreqs& freqs,
                             int32_t* positions_out, int32_t* dev_status, cudaStream_t stream);
}  // namespace ptd
