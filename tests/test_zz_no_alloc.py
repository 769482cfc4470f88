"""ptd_tree_attention_noalloc: the attention entry point for callers that cannot allocate
device memory (for example a plugin inside another runtime that owns every allocation, or a
decode loop that cannot afford cudaMalloc's implicit synchronisation).

It takes its key-split scratch from a fixed array the library keeps in device memory, so
its output must equal, bit for bit, that of ptd_tree_attention given a caller workspace, on
consecutive calls that reuse the array with the previous call's contents still in it.  This file is
collected last so a failure here never hides the other tests.
"""
import ctypes

import numpy as np
import pytest
import torch

import oracle
from paper_2607_10661_gb300 import ptd
from paper_2607_10661_gb300 import synthetic as syn
from paper_2607_10661_gb300.harness import DeviceWorkload

pytestmark = pytest.mark.gpu

BF16_MAX, BF16_MEAN = 2e-2, 2e-3
STATIC_SCRATCH_BYTES = 48 << 20    # PTD_STATIC_SCRATCH_BYTES in include/ptd.h


@pytest.fixture(scope="module", autouse=True)
def _built():
    import __graft_entry__

    __graft_entry__.build()


def _noalloc(dw, out):
    c = dw.w.cfg
    return ptd.lib().ptd_tree_attention_noalloc(
        ctypes.byref(dw.tree.c), ctypes.byref(dw.cache.c), 0, c.layers, dw.q.data_ptr(), c.hq, ctypes.c_float(0.0),
        out.data_ptr(), dw.dev_status.data_ptr(), ctypes.c_void_p(torch.cuda.current_stream().cuda_stream))


def _case(cfg_name, seed, **over):
    w = syn.Workload(syn.shrink(syn.CONFIGS[cfg_name], **over), seed)
    dw = DeviceWorkload(w, with_step_buffers=False)
    need = ptd.attention_workspace_size(dw.tree, dw.cache, w.cfg.hq)
    return dw, need


def test_noalloc_matches_workspace_entry_on_consecutive_calls():
    """Bit-identical to the workspace call (the same kernel and schedule, and the merge of a
    unit's pieces runs in a fixed order), on two calls in a row per shape and across shapes,
    so nothing left in the shared array by one call leaks into the next; the first case (a long
    context over few KV heads: the balanced schedule, units cut into pieces whose partials go
    through the array) is also checked against the oracle."""
    cases = [
        _case("long-context", 71, ctx=(3000, 3000), vocab=100),
        _case("llama2-7b-layer", 72, hq=8, hkv=8, ctx=(333, 333), vocab=100),
        _case("batched-paged", 73, batch=2, ctx=(300, 600), vocab=100, hq=8, hkv=2),
    ]
    for dw, need in cases:
        assert 0 < need <= STATIC_SCRATCH_BYTES, need
    assert cases[0][1] > (32 << 20)                       # the partials of one CTA per SM
    for dw, _ in cases:
        dw.dev_status.zero_()
        ref = torch.zeros_like(dw.q)
        dw.attn_out = ref
        dw.attention()                                    # ptd_tree_attention with a workspace
        for call in range(2):                             # two calls in a row on the shared array
            got = torch.full_like(dw.q, float("nan"))
            assert _noalloc(dw, got) == ptd.OK
            torch.cuda.synchronize()
            assert int(dw.dev_status.item()) == 0
            assert torch.equal(got, ref), call
    dw, _ = cases[0]
    w = dw.w
    got = dw.attn_out.float().cpu().numpy()
    q = syn.widen(w.q_layer(0), "bf16")
    kc, vc = (syn.widen(x, "bf16") for x in w.kv_layer(0))
    o = oracle.tree_attention(q, w.seq_view(kc, 0), w.seq_view(vc, 0), w.trees[0], int(w.ctx_lens[0]))
    err = np.abs(got[0] - o)
    assert err.max() <= BF16_MAX and err.mean() <= BF16_MEAN


def test_noalloc_rejects_problems_beyond_its_scratch():
    """Shapes whose scratch exceeds the array (here 262144 (tree, KV head, M-tile pair) units:
    their piece counters alone take 16 MB) are refused before anything is enqueued; the tree and
    cache descriptions point at no memory the call may touch."""
    A = 1 << 24
    t = ptd._Tree(8192, 8192, 128, 100, A, A + 65536, A + 131072)
    c = ptd._Cache(A * 2, A * 4, ptd.BF16, 1, 8, 128, 0, 1024, 0, None, 0)
    need = ptd.lib().ptd_attention_workspace_size(ctypes.byref(t), ctypes.byref(c), 64, 1)
    assert need > STATIC_SCRATCH_BYTES, need
    st = ptd.lib().ptd_tree_attention_noalloc(ctypes.byref(t), ctypes.byref(c), 0, 1, A * 8, 64, ctypes.c_float(0.0),
                                             A * 16, A * 32, ctypes.c_void_p(torch.cuda.current_stream().cuda_stream))
    assert st == ptd.WORKSPACE
