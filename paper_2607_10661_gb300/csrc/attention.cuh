// Internal launch parameters of the tree-attention kernels (not part of the C ABI).
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>

#include <cstddef>
#include <cstdint>

namespace ptd {

struct AttnParams {
  const void* q;               // [layers][n_total][hq][D]
  void* out;                   // [layers][n_total][hq][D]
  float* part_o;               // split partials: [units][splits][256][D] fp32
  float* part_ml;              // [units][splits][256][2] (running max in log2 units, sum)
  const int32_t* node_offsets;
  const int32_t* parents;
  const int32_t* ctx_lens;
  const int32_t* block_table;
  const void* k;               // cache base pointers (SIMT path)
  const void* v;
  int32_t* dev_status;
  int batch, hq, hkv, group, head_dim;
  int layer_begin, layers;     // layers of this call
  int n_total, max_nodes;
  int pairs;                   // 256-row M-tile pairs per (tree, KV head)
  int splits;                  // KV splits
  int page_size, seq_capacity, num_pages, max_pages;
  float scale_log2;            // scale * log2(e)
  float scale;
};

size_t tc_smem_bytes();
cudaError_t launch_tree_attn_tc(const CUtensorMap& map_k, const CUtensorMap& map_v, const AttnParams& p,
                                int units, cudaStream_t stream);
cudaError_t launch_attn_combine(const AttnParams& p, int units, cudaStream_t stream);
cudaError_t launch_tree_attn_simt(const AttnParams& p, cudaStream_t stream);

}  // namespace ptd
