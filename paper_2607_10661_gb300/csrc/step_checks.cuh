// Internal (not part of the C ABI): the host checks of one tree-verify step's arguments,
// shared by the entry points that enqueue work for a step before they run it.
#pragma once
#include "../../include/ptd.h"

namespace ptd {
// PTD_OK when ptd_tree_verify_step would pass its top-k and verification + compaction
// checks with these arguments (and q and logits are given); touches no device state.
ptd_status check_step_args(const ptd_tree* tree, const ptd_kv_cache* cache, const ptd_step_args* a);
}  // namespace ptd
