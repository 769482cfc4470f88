"""PTD tree-verify step on one GB300 (sm_103a): tree attention, per-node top-k, greedy
verification and KV compaction as hand-written CUDA kernels behind a C ABI (libptd.so).

`ptd` is the Python binding (argument marshalling only); `synthetic` draws seeded inputs.
"""
from . import ptd  # noqa: F401
from .ptd import (  # noqa: F401
    KVCache,
    PtdError,
    StepBuffers,
    Tree,
    attention_workspace_size,
    kv_compact,
    topk_draft,
    tree_attention,
    tree_verify_step,
    tree_verify_step_host,
    verify_greedy,
)
