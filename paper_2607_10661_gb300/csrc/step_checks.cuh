// Internal (not part of the C ABI): the host checks of one tree-verify step's arguments,
// shared by the entry points that enqueue work for a step before they run it.
#pragma once
#include "../../include/ptd.h"

namespace ptd {
// PTD_OK when ptd_tree_verify_step would pass its top-k and verification + compaction
// checks with these arguments (and q and logits are given); touches no device state.
ptd_status check_step_args(const ptd_tree* tree, const ptd_kv_cache* cache, const ptd_step_args* a);
// PTD_OK when the host copies of a step's tree layout describe `tree` and fit the cache:
// node_offsets_h[0] = 0, every tree has 1 .. max_nodes nodes, node_offsets_h[B] =
// total_nodes, and every context C >= 0 with C + T <= seq_capacity (contiguous) or
// max_pages * page_size (paged).  Reads host memory only.
ptd_status check_host_tree_layout(const ptd_tree* tree, const ptd_kv_cache* cache, const int32_t* node_offsets_h,
                                  const int32_t* ctx_lens_h);
}  // namespace ptd
