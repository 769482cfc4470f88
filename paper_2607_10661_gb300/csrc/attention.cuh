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
  float* part_o;               // piece partials: [slot][M tile][D / 4][128 rows][4] fp32 (O unnormalised)
  float* part_ml;              // [slot][256 rows][2] (running max in log2 units, row sum)
  unsigned long long* counters;   // persistent schedule: pieces finished per (unit, 32-row block):
                                  // (epoch << 32) | count, a value of another epoch counting as 0
  uint32_t epoch;                 // this launch's epoch (never 0)
  unsigned int* zero_ptr;         // zero_count words that CTA 0 clears after its dependency wait:
  int zero_count;                 // the step's tail counters, read by the kernels after this one
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
  int persistent;              // 1: balanced persistent schedule, one CTA per SM
  int defer_merge;             // persistent: every piece leaves a partial; tree_attn_merge_kernel merges
  int ctas;                    // persistent: the attention grid's CTAs (the cut the merge kernel follows)
  int q_tma;                   // 1: Q tiles arrive by TMA (map_q), else by per-thread loads
  int page_size, seq_capacity, num_pages, max_pages;
  float scale_log2;            // scale * log2(e)
  float scale;
};

size_t tc_smem_bytes();
// Launched with programmatic stream serialization: the kernel's set-up (barriers, tensor
// memory, descriptor prefetch) may overlap the stream's previous grid; it waits for that grid
// before its first global access.
cudaError_t launch_tree_attn_tc(const CUtensorMap& map_k, const CUtensorMap& map_v, const CUtensorMap& map_q,
                                const AttnParams& p, dim3 grid, cudaStream_t stream);
cudaError_t launch_tree_attn_simt(const AttnParams& p, cudaStream_t stream);
// The merge of the units the persistent cut split, after the attention kernel (programmatic
// dependent launch): one CTA per unit, the pieces' partials combined in CTA order.
cudaError_t launch_tree_attn_merge(const AttnParams& p, int units, int sms, cudaStream_t stream);

}  // namespace ptd
