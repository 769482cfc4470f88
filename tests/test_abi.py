"""The C ABI library builds, loads and exports every function include/ptd.h declares;
host-side argument checks reject bad calls before touching the GPU (no GPU needed)."""
import ctypes
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def lib():
    import __graft_entry__
    from paper_2607_10661_gb300 import ptd

    __graft_entry__.build()
    return ptd.lib()


def _declared_functions():
    src = open(os.path.join(ROOT, "include", "ptd.h")).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(ptd_[a-z_0-9]+)\s*\(", src)))


def test_header_declares_the_four_steps():
    names = _declared_functions()
    for n in ("ptd_tree_attention", "ptd_topk_draft", "ptd_verify_greedy", "ptd_kv_compact"):
        assert n in names


def test_every_declared_symbol_is_exported(lib):
    from paper_2607_10661_gb300 import ptd

    names = _declared_functions()
    assert names, "no declarations parsed"
    for n in names:
        assert hasattr(lib, n), n
    assert set(names) == set(ptd.EXPORTED)


def test_status_strings(lib):
    from paper_2607_10661_gb300 import ptd

    for s in range(8):
        assert ptd.status_string(s) and ptd.status_string(s) != "unknown status"
    assert ptd.status_string(0) == "ok"


def test_host_checks_reject_without_gpu(lib):
    from paper_2607_10661_gb300 import ptd

    null = ctypes.c_void_p(0)
    assert lib.ptd_topk_draft(null, ptd.BF16, 4, 100, 100, 2, null, null, null) == ptd.INVALID_ARG
    assert lib.ptd_tree_attention(None, None, 0, 1, null, 8, 0.0, null, null, 0, null, null) == ptd.INVALID_ARG
    assert lib.ptd_verify_greedy(None, null, null, 1, null, null, null, null, null) == ptd.INVALID_ARG
    assert lib.ptd_kv_compact(None, None, null, null, null, null) == ptd.INVALID_ARG
    assert lib.ptd_verify_and_compact(None, None, null, null, 1, null, null, null, null, null, null) == ptd.INVALID_ARG
    t1 = ptd._Tree(1, 10, 10, 0, 8, 8, 8)
    assert lib.ptd_verify_sampling(ctypes.byref(t1), 16, 16, ptd.BF16, 100, 100, 0.0, 16, 16, 16, 16, 16, 16,
                                   None) == ptd.INVALID_ARG   # temperature must be > 0
    assert lib.ptd_verify_sampling(ctypes.byref(t1), 16, None, ptd.BF16, 100, 100, 1.0, 16, 16, 16, 16, 16, 16,
                                   None) == ptd.INVALID_ARG
    # draft tree update: capacity above 128, expand above the draft row, aliased output, null pointer
    du = lambda **k: lib.ptd_draft_tree_update(
        k.get("batch", 1), 8, 16, k.get("inp", 32), 48, 64, k.get("dstride", 4), k.get("expand", 1), 4,
        k.get("max_depth", 6), k.get("capacity", 64), 80, k.get("outp", 96), 112, 128, 144, k.get("status", 160),
        None)
    assert du(capacity=129) == ptd.INVALID_ARG
    assert du(capacity=0) == ptd.INVALID_ARG
    assert du(expand=5, dstride=4) == ptd.INVALID_ARG
    assert du(expand=17, dstride=32) == ptd.INVALID_ARG
    assert du(max_depth=0) == ptd.INVALID_ARG
    assert du(batch=0) == ptd.INVALID_ARG
    assert du(outp=32) == ptd.INVALID_ARG
    assert du(status=None) == ptd.INVALID_ARG
    # candidate pool: capacity not a power of two, width above the kept children, bad budgets
    assert lib.ptd_pool_bytes(1000) == 0 and lib.ptd_pool_bytes(1 << 20) > (1 << 20) * 48
    assert lib.ptd_pool_init(None, 1024, None) == ptd.INVALID_ARG
    assert lib.ptd_pool_init(16, 1000, None) == ptd.INVALID_ARG
    assert lib.ptd_pool_merge(16, 1024, 2048, 0, 16, 16, 16, 16, None) == ptd.INVALID_ARG     # max_load > capacity
    assert lib.ptd_pool_merge(16, 1024, 512, -1, 16, 16, 16, 16, None) == ptd.INVALID_ARG    # negative step
    assert lib.ptd_pool_retrieve(16, 1024, 16, 9, 4, 64, 16, 16, 16, None) == ptd.INVALID_ARG  # width > 8
    assert lib.ptd_pool_retrieve(16, 1024, 16, 4, 0, 64, 16, 16, 16, None) == ptd.INVALID_ARG  # max_depth 0
    assert lib.ptd_pool_retrieve(16, 1024, 16, 4, 4, 129, 16, 16, 16, None) == ptd.INVALID_ARG  # max_nodes > 128
    # tree positions / rotary encoding: no tree, layer range past the cache, odd head_dim, base <= 1
    assert lib.ptd_tree_rope_append(None, None, 0, 1, 16, 32, 16, 16, 10000.0, None, 16, None) == ptd.INVALID_ARG
    tr_ = ptd._Tree(1, 10, 10, 0, 16, 16, 16)
    cr = ptd._Cache(16, 16, ptd.BF16, 2, 8, 128, 0, 300, 0, None, 0)
    assert lib.ptd_tree_rope_append(ctypes.byref(tr_), ctypes.byref(cr), 1, 2, 16, 32, 16, 16, 10000.0, None, 16,
                                    None) == ptd.INVALID_ARG
    assert lib.ptd_tree_rope_append(ctypes.byref(tr_), ctypes.byref(cr), 0, 1, 16, 32, 16, 16, 1.0, None, 16,
                                    None) == ptd.INVALID_ARG
    assert lib.ptd_tree_rope_append(ctypes.byref(tr_), ctypes.byref(cr), 0, 1, 16, 12, 16, 16, 1e4, None, 16,
                                    None) == ptd.INVALID_ARG     # 12 query heads over 8 KV heads
    t = ptd._Tree(1, 200, 200, 0, 8, 8, 8)          # max_nodes above 128
    c = ptd._Cache(16, 16, ptd.BF16, 1, 8, 128, 0, 300, 0, None, 0)
    assert lib.ptd_tree_attention(ctypes.byref(t), ctypes.byref(c), 0, 1, 16, 32, 0.0, 16, None, 0, 16,
                                  None) == ptd.INVALID_ARG
    t = ptd._Tree(1, 10, 10, 0, 8, 8, 8)
    c = ptd._Cache(16, 16, ptd.BF16, 1, 8, 128, 24, 0, 4, 8, 4)   # page size 24 is not supported
    assert lib.ptd_tree_attention(ctypes.byref(t), ctypes.byref(c), 0, 1, 16, 32, 0.0, 16, None, 0, 16,
                                  None) == ptd.UNSUPPORTED
    assert lib.ptd_attention_workspace_size(ctypes.byref(t), ctypes.byref(c), 32, 1) == 0


def test_binding_rejects_host_tensors_and_bad_dtypes(lib):
    """The Python binding checks device, layout and dtype before any call into the library:
    there is no host fallback, a CPU tensor is an error."""
    import torch
    from paper_2607_10661_gb300 import ptd

    logits = torch.zeros((4, 100), dtype=torch.bfloat16)
    idx = torch.zeros((4, 2), dtype=torch.int32)
    val = torch.zeros((4, 2), dtype=torch.float32)
    with pytest.raises(ValueError, match="CUDA tensor"):
        ptd.topk_draft(logits, 2, idx, val)
    with pytest.raises(TypeError):
        ptd._dev([1, 2, 3], "x")
    with pytest.raises(ValueError, match="contiguous host"):
        ptd._host(torch.zeros((4, 4)).t(), "x")
    with pytest.raises(TypeError):
        ptd._host(torch.zeros(4, dtype=torch.int64), "x", torch.int32)
    with pytest.raises(TypeError, match="unsupported dtype"):
        ptd._ptd_dtype(torch.float16)


def test_missing_library_fails_loudly(monkeypatch):
    """Without the built library every entry point raises: nothing falls back to the host."""
    from paper_2607_10661_gb300 import ptd

    monkeypatch.setattr(ptd, "_lib", None)
    monkeypatch.setattr(ptd, "LIB_PATH", os.path.join(ROOT, "no-such-dir", "libptd.so"))
    with pytest.raises(RuntimeError, match="not built"):
        ptd.lib()


def _step_structs(ptd, **kw):
    """A Llama-3-8B-shaped step description over fake, aligned device addresses: the host
    checks read only the sizes and the pointers' presence and alignment."""
    A = 1 << 20
    t = ptd._Tree(1, 63, 63, 8192, A, A + 1024, A + 2048)
    c = ptd._Cache(A * 2, A * 4, ptd.BF16, 32, 8, 128, 0, 8320, 0, None, 0)
    d = dict(q=A * 8, num_q_heads=32, scale=0.0, attn_out=A * 16, logits=A * 32, logits_dtype=ptd.BF16,
             vocab=128256, k=4, tokens=A + 4096, topk_idx=A + 8192, topk_val=A + 12288, accepted_nodes=A + 16384,
             accept_len=A + 20480, bonus_token=A + 20544, new_ctx_lens=A + 20608, dev_status=A + 20672,
             workspace=None, workspace_bytes=0)
    d.update(kw)
    return t, c, ptd._StepArgs(**d)


def _no_cuda():
    import torch

    return not torch.cuda.is_available()


# Host-logic checks on fake device addresses: they run only where no GPU is visible.
host_only = pytest.mark.skipif(not _no_cuda(), reason="host-side checks with fake device addresses")


@host_only
@pytest.mark.parametrize("bad", [dict(k=0), dict(k=17), dict(logits=None), dict(logits_dtype=7), dict(tokens=None),
                                 dict(new_ctx_lens=(1 << 20) + 2048), dict(dev_status=None), dict(topk_idx=None)])
def test_step_checks_every_part_before_the_first_launch(lib, bad):
    """ptd_tree_verify_step rejects a bad argument of its top-k or verification part before
    it launches the attention (whose own checks would pass here): the call returns
    INVALID_ARG, not the CUDA error that any launch attempt gives on a machine without a GPU."""
    from paper_2607_10661_gb300 import ptd

    t, c, a = _step_structs(ptd, **bad)
    assert lib.ptd_tree_verify_step(ctypes.byref(t), ctypes.byref(c), ctypes.byref(a), None) == ptd.INVALID_ARG


@host_only
def test_host_step_checks_before_the_first_copy(lib):
    """ptd_tree_verify_step_host rejects bad step arguments and a tree that does not fit the
    cache before it enqueues any copy (no CUDA call is reached here)."""
    import numpy as np
    from paper_2607_10661_gb300 import ptd

    offs = np.array([0, 63], np.int32)
    ctx = np.array([8192], np.int32)
    fake = 1 << 24
    io = ptd._HostIO(*([fake] * 4 + [offs.ctypes.data, ctx.ctypes.data] + [fake] * 9))
    t, c, a = _step_structs(ptd, k=0)
    assert lib.ptd_tree_verify_step_host(ctypes.byref(t), ctypes.byref(c), ctypes.byref(a), ctypes.byref(io),
                                         None) == ptd.INVALID_ARG
    t, c, a = _step_structs(ptd, q=None)
    assert lib.ptd_tree_verify_step_host(ctypes.byref(t), ctypes.byref(c), ctypes.byref(a), ctypes.byref(io),
                                         None) == ptd.INVALID_ARG
    ctx[0] = 8300                     # 8300 + 63 slots > the cache's 8320
    t, c, a = _step_structs(ptd)
    assert lib.ptd_tree_verify_step_host(ctypes.byref(t), ctypes.byref(c), ctypes.byref(a), ctypes.byref(io),
                                         None) == ptd.INVALID_ARG


@host_only
@pytest.mark.parametrize("bad", [dict(k=0), dict(logits=None), dict(q=None), dict(new_ctx_lens=(1 << 20) + 2048)])
def test_pipeline_create_checks_the_step_arguments(lib, bad):
    """ptd_pipeline_create runs the step's checks on both slots' arguments before it creates
    anything, so a bad argument cannot surface later with uploads already enqueued."""
    from paper_2607_10661_gb300 import ptd

    t0, c, a0 = _step_structs(ptd)
    t1, _, a1 = _step_structs(ptd, **bad)
    trees = (ptd._Tree * 2)(t0, t1)
    args = (ptd._StepArgs * 2)(a0, a1)
    staging = (ctypes.c_void_p * 2)(1 << 26, 1 << 27)
    out = ctypes.c_void_p(0)
    st = lib.ptd_pipeline_create(ctypes.byref(c), trees, args, staging, 1 << 40, None, ctypes.byref(out))
    assert st == ptd.INVALID_ARG and not out.value
    # the same description with good arguments in both slots passes the checks and gets as
    # far as creating the pipeline's streams, which fails here only because there is no GPU
    trees = (ptd._Tree * 2)(t0, t0)
    args = (ptd._StepArgs * 2)(a0, a0)
    st = lib.ptd_pipeline_create(ctypes.byref(c), trees, args, staging, 1 << 40, None, ctypes.byref(out))
    assert st == ptd.CUDA_ERROR and not out.value


@host_only
@pytest.mark.parametrize("offs,ctx", [([1, 63], [8192]), ([0, 62], [8192]), ([0, 64], [8192]), ([0, 63], [-1]),
                                      ([0, 0], [8192])])
def test_host_step_rejects_a_bad_host_tree_layout(lib, offs, ctx):
    """A host offset array that does not describe the tree (not starting at 0, not ending at
    total_nodes, an empty tree) or a negative context is rejected before any copy: the host
    step would otherwise read the tree K/V rows past the host buffers."""
    import numpy as np
    from paper_2607_10661_gb300 import ptd

    o = np.array(offs, np.int32)
    cx = np.array(ctx, np.int32)
    fake = 1 << 24
    io = ptd._HostIO(*([fake] * 4 + [o.ctypes.data, cx.ctypes.data] + [fake] * 9))
    t, c, a = _step_structs(ptd)
    assert lib.ptd_tree_verify_step_host(ctypes.byref(t), ctypes.byref(c), ctypes.byref(a), ctypes.byref(io),
                                         None) == ptd.INVALID_ARG


@host_only
def test_host_step_rejects_a_tree_above_max_nodes(lib):
    """Two trees whose offsets add up to total_nodes but one of which exceeds max_nodes."""
    import numpy as np
    from paper_2607_10661_gb300 import ptd

    o = np.array([0, 40, 63], np.int32)
    cx = np.array([100, 100], np.int32)
    fake = 1 << 24
    io = ptd._HostIO(*([fake] * 4 + [o.ctypes.data, cx.ctypes.data] + [fake] * 9))
    A = 1 << 20
    t = ptd._Tree(2, 63, 32, 100, A, A + 1024, A + 2048)           # max_nodes 32 < 40
    _, c, a = _step_structs(ptd)
    assert lib.ptd_tree_verify_step_host(ctypes.byref(t), ctypes.byref(c), ctypes.byref(a), ctypes.byref(io),
                                         None) == ptd.INVALID_ARG


def test_step_topk_policy_round_trip(lib):
    """ptd_step_topk_policy (host only): each known policy is taken and the previous one is
    returned; an unknown one changes nothing and returns -1."""
    lib.ptd_step_topk_policy.restype = ctypes.c_int32
    lib.ptd_step_topk_policy.argtypes = [ctypes.c_int32]
    start = lib.ptd_step_topk_policy(0)
    try:
        assert lib.ptd_step_topk_policy(2) == 0
        assert lib.ptd_step_topk_policy(1) == 2
        assert lib.ptd_step_topk_policy(7) == -1
        assert lib.ptd_step_topk_policy(-1) == -1
        assert lib.ptd_step_topk_policy(0) == 1
    finally:
        lib.ptd_step_topk_policy(start)


@host_only
def test_step_tail_choice(lib):
    """ptd_step_tail (host only) gives the tail ptd_tree_verify_step would run: the clustered
    top-k for a one-wave step (63 rows of 128256), the streamed one for more than one wave
    (266 rows), either when forced, the clustered one where streaming cannot apply (vocab not a
    multiple of 8, logits off 16 bytes, a workspace holding only the per-tree counters), the
    separate verification without a workspace or with fp32 logits, and -1 for a missing tree."""
    from paper_2607_10661_gb300 import ptd

    A = 1 << 20

    def tail(tree=None, **kw):
        t, c, a = _step_structs(ptd, **kw)
        if tree is not None:
            t = tree
        return lib.ptd_step_tail(ctypes.byref(t), ctypes.byref(c), ctypes.byref(a)), t, c

    _, t, c = tail()
    full = lib.ptd_step_workspace_size(ctypes.byref(t), ctypes.byref(c), 32)
    attn = lib.ptd_attention_workspace_size(ctypes.byref(t), ctypes.byref(c), 32, 32)
    ws = dict(workspace=A * 64, workspace_bytes=full)
    assert tail()[0] == ptd.STEP_TAIL_SEPARATE
    assert tail(**ws)[0] == ptd.STEP_TAIL_CLUSTERED
    many = ptd._Tree(8, 266, 64, 4096, A, A + 1024, A + 2048)
    full_many = lib.ptd_step_workspace_size(ctypes.byref(many), ctypes.byref(c), 32)
    assert tail(many, workspace=A * 64, workspace_bytes=full_many)[0] == ptd.STEP_TAIL_STREAMED
    prev = ptd.step_topk_policy(ptd.STEP_TOPK_STREAMED)
    try:
        assert tail(**ws)[0] == ptd.STEP_TAIL_STREAMED
        assert tail(vocab=128250, **ws)[0] == ptd.STEP_TAIL_CLUSTERED
        assert tail(logits=A * 32 + 8, **ws)[0] == ptd.STEP_TAIL_CLUSTERED
        counters_only = (attn + 255) // 256 * 256 + 256
        assert tail(workspace=A * 64, workspace_bytes=counters_only)[0] == ptd.STEP_TAIL_CLUSTERED
        ptd.step_topk_policy(ptd.STEP_TOPK_CLUSTERED)
        assert tail(many, workspace=A * 64, workspace_bytes=full_many)[0] == ptd.STEP_TAIL_CLUSTERED
    finally:
        ptd.step_topk_policy(prev)
    assert tail(logits_dtype=ptd.F32, **ws)[0] == ptd.STEP_TAIL_SEPARATE
    t, c, a = _step_structs(ptd)
    assert lib.ptd_step_tail(None, ctypes.byref(c), ctypes.byref(a)) == -1
