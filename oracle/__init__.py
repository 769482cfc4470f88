"""CPU oracle of the PTD tree-verify step.

Test infrastructure: only the tests, `__graft_entry__.smoke()` and `bench.py`'s
CPU-baseline / reference arm may import it.  The product path never does.
"""
from .ptd_oracle import (  # noqa: F401
    CandidatePool,
    InvalidTree,
    ancestor_sets,
    check_forest,
    check_tree,
    children_sets,
    depths,
    draft_tree_update,
    eligible_edges,
    kv_compact,
    lm_head_logits,
    lm_head_topk,
    softmax_row,
    topk,
    topk_rows,
    tree_positions,
    rope,
    tree_attention,
    verify_greedy,
    verify_sampling,
    visibility,
)
