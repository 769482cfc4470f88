"""Python binding of libptd.so (the PTD tree-verify step C ABI, include/ptd.h).

Argument marshalling only: every function checks dtype / device / contiguity of the torch
tensors it is given, passes their data pointers and the current CUDA stream to the C ABI
function of the same name, and raises PtdError on a non-OK status.  All compute happens
in the CUDA kernels; there is no CPU path.  The library is loaded on first use and a
missing or unloadable libptd.so raises immediately.
"""
from __future__ import annotations

import ctypes
import os
from typing import Optional

import torch

_PKG = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_PKG, "libptd.so")

OK, INVALID_ARG, INVALID_TREE, UNSUPPORTED, CUDA_ERROR, TIMEOUT, WORKSPACE, POOL_FULL = range(8)
F32, BF16 = 0, 1
MAX_TREE_NODES = 128
MAX_TOPK = 16
MAX_EXPAND = 16
POOL_KIDS = 8

EXPORTED = (
    "ptd_attention_workspace_size", "ptd_tree_attention", "ptd_topk_draft", "ptd_verify_greedy",
    "ptd_kv_compact", "ptd_tree_verify_step", "ptd_tree_verify_step_host", "ptd_last_launch_count",
    "ptd_status_string", "ptd_tree_attention_noalloc", "ptd_verify_and_compact", "ptd_verify_sampling",
    "ptd_draft_tree_update", "ptd_pool_bytes", "ptd_pool_init", "ptd_pool_merge", "ptd_pool_retrieve",
    "ptd_tree_rope_append", "ptd_lm_head_topk_workspace_size", "ptd_lm_head_topk", "ptd_pipeline_create",
    "ptd_pipeline_submit", "ptd_pipeline_wait", "ptd_pipeline_destroy", "ptd_check_bounded_wait",
    "ptd_step_workspace_size", "ptd_step_topk_policy", "ptd_step_tail",
)


class PtdError(RuntimeError):
    def __init__(self, status: int, where: str):
        self.status = status
        super().__init__(f"{where}: {status_string(status)} (status {status})")


class _Tree(ctypes.Structure):
    _fields_ = [("batch", ctypes.c_int32), ("total_nodes", ctypes.c_int32), ("max_nodes", ctypes.c_int32),
                ("max_ctx", ctypes.c_int32), ("node_offsets", ctypes.c_void_p), ("parents", ctypes.c_void_p),
                ("ctx_lens", ctypes.c_void_p)]


class _Cache(ctypes.Structure):
    _fields_ = [("k", ctypes.c_void_p), ("v", ctypes.c_void_p), ("dtype", ctypes.c_int),
                ("num_layers", ctypes.c_int32), ("num_kv_heads", ctypes.c_int32), ("head_dim", ctypes.c_int32),
                ("page_size", ctypes.c_int32), ("seq_capacity", ctypes.c_int32), ("num_pages", ctypes.c_int32),
                ("block_table", ctypes.c_void_p), ("max_pages", ctypes.c_int32)]


class _StepArgs(ctypes.Structure):
    _fields_ = [("q", ctypes.c_void_p), ("num_q_heads", ctypes.c_int32), ("scale", ctypes.c_float),
                ("attn_out", ctypes.c_void_p), ("logits", ctypes.c_void_p), ("logits_dtype", ctypes.c_int),
                ("vocab", ctypes.c_int32), ("k", ctypes.c_int32), ("tokens", ctypes.c_void_p),
                ("topk_idx", ctypes.c_void_p), ("topk_val", ctypes.c_void_p), ("accepted_nodes", ctypes.c_void_p),
                ("accept_len", ctypes.c_void_p), ("bonus_token", ctypes.c_void_p),
                ("new_ctx_lens", ctypes.c_void_p), ("dev_status", ctypes.c_void_p), ("workspace", ctypes.c_void_p),
                ("workspace_bytes", ctypes.c_size_t)]


class _HostIO(ctypes.Structure):
    _fields_ = [(n, ctypes.c_void_p) for n in (
        "q_h", "logits_h", "tokens_h", "parents_h", "node_offsets_h", "ctx_lens_h", "tree_k_h", "tree_v_h",
        "topk_idx_h", "topk_val_h", "accepted_h", "accept_len_h", "bonus_h", "new_ctx_h", "status_h")]


_lib = None


def lib() -> ctypes.CDLL:
    """The loaded libptd.so (raises if it was not built)."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise RuntimeError(f"libptd.so not built ({LIB_PATH}); run __graft_entry__.build()")
        L = ctypes.CDLL(LIB_PATH)
        vp, i32, i64, f32, sz = ctypes.c_void_p, ctypes.c_int32, ctypes.c_int64, ctypes.c_float, ctypes.c_size_t
        P = ctypes.POINTER
        L.ptd_status_string.restype = ctypes.c_char_p
        L.ptd_status_string.argtypes = [ctypes.c_int]
        L.ptd_last_launch_count.restype = i32
        L.ptd_last_launch_count.argtypes = []
        L.ptd_step_topk_policy.restype = i32
        L.ptd_step_topk_policy.argtypes = [i32]
        L.ptd_step_tail.restype = i32
        L.ptd_step_tail.argtypes = [P(_Tree), P(_Cache), P(_StepArgs)]
        L.ptd_attention_workspace_size.restype = sz
        L.ptd_attention_workspace_size.argtypes = [P(_Tree), P(_Cache), i32, i32]
        L.ptd_step_workspace_size.restype = sz
        L.ptd_step_workspace_size.argtypes = [P(_Tree), P(_Cache), i32]
        L.ptd_tree_attention.restype = ctypes.c_int
        L.ptd_tree_attention.argtypes = [P(_Tree), P(_Cache), i32, i32, vp, i32, f32, vp, vp, sz, vp, vp]
        L.ptd_tree_attention_noalloc.restype = ctypes.c_int
        L.ptd_tree_attention_noalloc.argtypes = [P(_Tree), P(_Cache), i32, i32, vp, i32, f32, vp, vp, vp]
        L.ptd_topk_draft.restype = ctypes.c_int
        L.ptd_topk_draft.argtypes = [vp, ctypes.c_int, i64, i32, i64, i32, vp, vp, vp]
        L.ptd_verify_greedy.restype = ctypes.c_int
        L.ptd_verify_greedy.argtypes = [P(_Tree), vp, vp, i32, vp, vp, vp, vp, vp]
        L.ptd_kv_compact.restype = ctypes.c_int
        L.ptd_kv_compact.argtypes = [P(_Tree), P(_Cache), vp, vp, vp, vp]
        L.ptd_verify_sampling.restype = ctypes.c_int
        L.ptd_verify_sampling.argtypes = [P(_Tree), vp, vp, ctypes.c_int, i32, i64, f32, vp, vp, vp, vp, vp, vp, vp]
        L.ptd_verify_and_compact.restype = ctypes.c_int
        L.ptd_verify_and_compact.argtypes = [P(_Tree), P(_Cache), vp, vp, i32, vp, vp, vp, vp, vp, vp]
        L.ptd_draft_tree_update.restype = ctypes.c_int
        L.ptd_draft_tree_update.argtypes = [i32, i32, vp, vp, vp, vp, i32, i32, i32, i32, i32, vp, vp, vp, vp, vp,
                                            vp, vp]
        L.ptd_pool_bytes.restype = sz
        L.ptd_pool_bytes.argtypes = [i32]
        L.ptd_pool_init.restype = ctypes.c_int
        L.ptd_pool_init.argtypes = [vp, i32, vp]
        L.ptd_pool_merge.restype = ctypes.c_int
        L.ptd_pool_merge.argtypes = [vp, i32, i32, i32, vp, vp, vp, vp, vp]
        L.ptd_pool_retrieve.restype = ctypes.c_int
        L.ptd_pool_retrieve.argtypes = [vp, i32, vp, i32, i32, i32, vp, vp, vp, vp]
        L.ptd_tree_rope_append.restype = ctypes.c_int
        L.ptd_tree_rope_append.argtypes = [P(_Tree), P(_Cache), i32, i32, vp, i32, vp, vp, f32, vp, vp, vp]
        L.ptd_lm_head_topk_workspace_size.restype = sz
        L.ptd_lm_head_topk_workspace_size.argtypes = [i32, i32]
        L.ptd_lm_head_topk.restype = ctypes.c_int
        L.ptd_lm_head_topk.argtypes = [vp, i32, i64, vp, i32, i64, i32, i32, vp, vp, vp, sz, vp, vp]
        L.ptd_pipeline_create.restype = ctypes.c_int
        L.ptd_pipeline_create.argtypes = [P(_Cache), P(_Tree), P(_StepArgs), P(vp), sz, vp, P(vp)]
        L.ptd_pipeline_submit.restype = ctypes.c_int
        L.ptd_pipeline_submit.argtypes = [vp, P(_HostIO), P(i64)]
        L.ptd_pipeline_wait.restype = ctypes.c_int
        L.ptd_pipeline_wait.argtypes = [vp, i64]
        L.ptd_pipeline_destroy.restype = ctypes.c_int
        L.ptd_pipeline_destroy.argtypes = [vp]
        L.ptd_check_bounded_wait.restype = ctypes.c_int
        L.ptd_check_bounded_wait.argtypes = [vp, vp]
        L.ptd_tree_verify_step.restype = ctypes.c_int
        L.ptd_tree_verify_step.argtypes = [P(_Tree), P(_Cache), P(_StepArgs), vp]
        L.ptd_tree_verify_step_host.restype = ctypes.c_int
        L.ptd_tree_verify_step_host.argtypes = [P(_Tree), P(_Cache), P(_StepArgs), P(_HostIO), vp]
        _lib = L
    return _lib


def status_string(status: int) -> str:
    return lib().ptd_status_string(int(status)).decode()


STEP_TOPK_AUTO, STEP_TOPK_CLUSTERED, STEP_TOPK_STREAMED = 0, 1, 2


def step_topk_policy(policy: int) -> int:
    """ptd_step_topk_policy: which top-k the one-call step uses (process-wide); returns the previous one."""
    prev = int(lib().ptd_step_topk_policy(int(policy)))
    if prev < 0:
        raise ValueError(f"unknown step top-k policy {policy}")
    return prev


STEP_TAIL_SEPARATE, STEP_TAIL_CLUSTERED, STEP_TAIL_STREAMED = 0, 1, 2


def step_tail(tree: Tree, cache: KVCache, bufs: "StepBuffers") -> int:
    """ptd_step_tail: which tail tree_verify_step would run (0 separate verify + compact,
    1 clustered top-k verifying, 2 streamed top-k verifying)."""
    t = int(lib().ptd_step_tail(ctypes.byref(tree.c), ctypes.byref(cache.c), ctypes.byref(bufs.c)))
    if t < 0:
        raise ValueError("ptd_step_tail: invalid tree, cache or step arguments")
    return t


def last_launch_count() -> int:
    """Kernels the last successful C-ABI call on this thread enqueued."""
    return int(lib().ptd_last_launch_count())


def _check(status: int, where: str) -> None:
    if status != OK:
        raise PtdError(status, where)


def _dev(t: torch.Tensor, name: str, dtype=None, row_strided: bool = False) -> int:
    """Device pointer of t; row_strided accepts a 2-D tensor whose rows are apart (unit column stride)."""
    if not isinstance(t, torch.Tensor):
        raise TypeError(f"{name} must be a torch.Tensor")
    if not t.is_cuda:
        raise ValueError(f"{name} must be a CUDA tensor")
    if row_strided:
        if t.dim() != 2 or t.stride(1) != 1 or t.stride(0) < t.shape[1]:
            raise ValueError(f"{name} must be [rows, cols] with unit column stride")
    elif not t.is_contiguous():
        raise ValueError(f"{name} must be contiguous")
    if dtype is not None and t.dtype != dtype:
        raise TypeError(f"{name} must be {dtype}, got {t.dtype}")
    return t.data_ptr()


def _host(t: torch.Tensor, name: str, dtype=None) -> int:
    if t.is_cuda or not t.is_contiguous():
        raise ValueError(f"{name} must be a contiguous host tensor")
    if dtype is not None and t.dtype != dtype:
        raise TypeError(f"{name} must be {dtype}, got {t.dtype}")
    return t.data_ptr()


def _ptd_dtype(dt: torch.dtype) -> int:
    if dt == torch.bfloat16:
        return BF16
    if dt == torch.float32:
        return F32
    raise TypeError(f"unsupported dtype {dt}")


def _stream(stream) -> int:
    if stream is None:
        stream = torch.cuda.current_stream()
    return int(stream.cuda_stream) if hasattr(stream, "cuda_stream") else int(stream)


class Tree:
    """A batch of trees in device memory (node_offsets [B+1], parents [N_tot], ctx_lens [B], int32)."""

    def __init__(self, node_offsets: torch.Tensor, parents: torch.Tensor, ctx_lens: torch.Tensor,
                 max_nodes: int, max_ctx: int):
        self.node_offsets, self.parents, self.ctx_lens = node_offsets, parents, ctx_lens
        self.batch = ctx_lens.numel()
        self.total_nodes = parents.numel()
        self.c = _Tree(self.batch, self.total_nodes, int(max_nodes), int(max_ctx),
                       _dev(node_offsets, "node_offsets", torch.int32), _dev(parents, "parents", torch.int32),
                       _dev(ctx_lens, "ctx_lens", torch.int32))


class KVCache:
    """K/V cache in device memory: contiguous [L][B][S_cap][Hkv][D] or paged [L][P][page][Hkv][D]."""

    def __init__(self, k: torch.Tensor, v: torch.Tensor, num_kv_heads: int, head_dim: int, page_size: int = 0,
                 block_table: Optional[torch.Tensor] = None):
        if k.shape != v.shape or k.dtype != v.dtype:
            raise ValueError("k and v must have the same shape and dtype")
        self.k, self.v, self.block_table = k, v, block_table
        self.num_layers = k.shape[0]
        self.num_kv_heads, self.head_dim, self.page_size = int(num_kv_heads), int(head_dim), int(page_size)
        if page_size:
            num_pages, seq_capacity = k.shape[1], 0
            max_pages = block_table.shape[1]
            bt = _dev(block_table, "block_table", torch.int32)
        else:
            num_pages, seq_capacity, max_pages, bt = 0, k.shape[2], 0, None
        self.c = _Cache(_dev(k, "k"), _dev(v, "v"), _ptd_dtype(k.dtype), self.num_layers, self.num_kv_heads,
                        self.head_dim, self.page_size, seq_capacity, num_pages, bt, max_pages)


def attention_workspace_size(tree: Tree, cache: KVCache, num_q_heads: int, num_layers: Optional[int] = None) -> int:
    n = cache.num_layers if num_layers is None else num_layers
    return int(lib().ptd_attention_workspace_size(ctypes.byref(tree.c), ctypes.byref(cache.c), num_q_heads, n))


def step_workspace_size(tree: Tree, cache: KVCache, num_q_heads: int) -> int:
    """ptd_step_workspace_size: the one-call step's scratch (attention's, then the tail's counters)."""
    return int(lib().ptd_step_workspace_size(ctypes.byref(tree.c), ctypes.byref(cache.c), num_q_heads))


def tree_attention(tree: Tree, cache: KVCache, q: torch.Tensor, out: torch.Tensor, num_q_heads: int,
                   dev_status: torch.Tensor, layer_begin: int = 0, num_layers: Optional[int] = None,
                   scale: float = 0.0, workspace: Optional[torch.Tensor] = None, stream=None) -> int:
    """ptd_tree_attention; returns the number of kernels launched."""
    n = cache.num_layers if num_layers is None else num_layers
    ws = _dev(workspace, "workspace") if workspace is not None else None
    wsb = workspace.numel() * workspace.element_size() if workspace is not None else 0
    st = lib().ptd_tree_attention(ctypes.byref(tree.c), ctypes.byref(cache.c), layer_begin, n,
                                  _dev(q, "q", cache.k.dtype), num_q_heads, float(scale),
                                  _dev(out, "out", cache.k.dtype), ws, wsb, _dev(dev_status, "dev_status", torch.int32),
                                  _stream(stream))
    _check(st, "ptd_tree_attention")
    return last_launch_count()


def topk_draft(logits: torch.Tensor, k: int, out_idx: torch.Tensor, out_val: torch.Tensor,
               vocab: Optional[int] = None, stream=None) -> int:
    """ptd_topk_draft over the rows of a 2-D logits tensor."""
    rows, stride = logits.shape
    st = lib().ptd_topk_draft(_dev(logits, "logits"), _ptd_dtype(logits.dtype), rows,
                              stride if vocab is None else vocab, stride, k,
                              _dev(out_idx, "out_idx", torch.int32), _dev(out_val, "out_val", torch.float32),
                              _stream(stream))
    _check(st, "ptd_topk_draft")
    return last_launch_count()


def verify_greedy(tree: Tree, tokens: torch.Tensor, target: torch.Tensor, target_stride: int,
                  accepted: torch.Tensor, accept_len: torch.Tensor, bonus: torch.Tensor, dev_status: torch.Tensor,
                  stream=None) -> int:
    st = lib().ptd_verify_greedy(ctypes.byref(tree.c), _dev(tokens, "tokens", torch.int32),
                                 _dev(target, "target", torch.int32), target_stride,
                                 _dev(accepted, "accepted", torch.int32), _dev(accept_len, "accept_len", torch.int32),
                                 _dev(bonus, "bonus", torch.int32), _dev(dev_status, "dev_status", torch.int32),
                                 _stream(stream))
    _check(st, "ptd_verify_greedy")
    return last_launch_count()


def kv_compact(tree: Tree, cache: KVCache, accepted: torch.Tensor, accept_len: torch.Tensor,
               new_ctx: torch.Tensor, stream=None) -> int:
    st = lib().ptd_kv_compact(ctypes.byref(tree.c), ctypes.byref(cache.c), _dev(accepted, "accepted", torch.int32),
                              _dev(accept_len, "accept_len", torch.int32), _dev(new_ctx, "new_ctx", torch.int32),
                              _stream(stream))
    _check(st, "ptd_kv_compact")
    return last_launch_count()


def verify_sampling(tree: Tree, tokens: torch.Tensor, logits: torch.Tensor, temperature: float,
                    u_accept: torch.Tensor, u_bonus: torch.Tensor, accepted: torch.Tensor, accept_len: torch.Tensor,
                    bonus: torch.Tensor, dev_status: torch.Tensor, stream=None) -> int:
    """ptd_verify_sampling; logits [N_tot, V] (bf16 or fp32), uniforms fp32."""
    if logits.dim() != 2 or logits.stride(1) != 1:
        raise ValueError("logits must be [rows, vocab] with unit column stride")
    dt = BF16 if logits.dtype == torch.bfloat16 else F32
    st = lib().ptd_verify_sampling(ctypes.byref(tree.c), _dev(tokens, "tokens", torch.int32),
                                   _dev(logits, "logits", logits.dtype, row_strided=True), dt, logits.shape[1],
                                   logits.stride(0),
                                   float(temperature), _dev(u_accept, "u_accept", torch.float32),
                                   _dev(u_bonus, "u_bonus", torch.float32), _dev(accepted, "accepted", torch.int32),
                                   _dev(accept_len, "accept_len", torch.int32), _dev(bonus, "bonus", torch.int32),
                                   _dev(dev_status, "dev_status", torch.int32), _stream(stream))
    _check(st, "ptd_verify_sampling")
    return last_launch_count()


def verify_and_compact(tree: Tree, cache: KVCache, tokens: torch.Tensor, target: torch.Tensor, target_stride: int,
                       accepted: torch.Tensor, accept_len: torch.Tensor, bonus: torch.Tensor, new_ctx: torch.Tensor,
                       dev_status: torch.Tensor, stream=None) -> int:
    st = lib().ptd_verify_and_compact(ctypes.byref(tree.c), ctypes.byref(cache.c), _dev(tokens, "tokens", torch.int32),
                                      _dev(target, "target", torch.int32), target_stride,
                                      _dev(accepted, "accepted", torch.int32),
                                      _dev(accept_len, "accept_len", torch.int32), _dev(bonus, "bonus", torch.int32),
                                      _dev(new_ctx, "new_ctx", torch.int32), _dev(dev_status, "dev_status", torch.int32),
                                      _stream(stream))
    _check(st, "ptd_verify_and_compact")
    return last_launch_count()


class StepBuffers:
    """Device buffers of one whole tree-verify step (inputs and outputs)."""

    def __init__(self, q, num_q_heads, attn_out, logits, k, tokens, topk_idx, topk_val, accepted, accept_len, bonus,
                 new_ctx, dev_status, workspace=None, scale=0.0):
        self.keep = (q, attn_out, logits, tokens, topk_idx, topk_val, accepted, accept_len, bonus, new_ctx,
                     dev_status, workspace)
        self.q, self.attn_out, self.logits, self.tokens = q, attn_out, logits, tokens
        self.topk_idx, self.topk_val, self.accepted, self.accept_len = topk_idx, topk_val, accepted, accept_len
        self.bonus, self.new_ctx, self.dev_status, self.workspace = bonus, new_ctx, dev_status, workspace
        self.k = int(k)
        self.c = _StepArgs(
            _dev(q, "q"), int(num_q_heads), float(scale), _dev(attn_out, "attn_out"), _dev(logits, "logits"),
            _ptd_dtype(logits.dtype), logits.shape[1], int(k), _dev(tokens, "tokens", torch.int32),
            _dev(topk_idx, "topk_idx", torch.int32), _dev(topk_val, "topk_val", torch.float32),
            _dev(accepted, "accepted", torch.int32), _dev(accept_len, "accept_len", torch.int32),
            _dev(bonus, "bonus", torch.int32), _dev(new_ctx, "new_ctx", torch.int32),
            _dev(dev_status, "dev_status", torch.int32),
            _dev(workspace, "workspace") if workspace is not None else None,
            workspace.numel() * workspace.element_size() if workspace is not None else 0)


def tree_verify_step(tree: Tree, cache: KVCache, bufs: StepBuffers, stream=None) -> int:
    """ptd_tree_verify_step: attention, top-k, verification and compaction on device buffers."""
    st = lib().ptd_tree_verify_step(ctypes.byref(tree.c), ctypes.byref(cache.c), ctypes.byref(bufs.c),
                                    _stream(stream))
    _check(st, "ptd_tree_verify_step")
    return last_launch_count()


class HostIO:
    """Pinned host tensors for ptd_tree_verify_step_host."""

    def __init__(self, **t):
        self.t = t
        self.c = _HostIO(*[_host(t[n], n) for n, _ in _HostIO._fields_])


def tree_verify_step_host(tree: Tree, cache: KVCache, bufs: StepBuffers, io: HostIO, stream=None) -> int:
    """ptd_tree_verify_step_host: host inputs -> device step -> host results (asynchronous)."""
    st = lib().ptd_tree_verify_step_host(ctypes.byref(tree.c), ctypes.byref(cache.c), ctypes.byref(bufs.c),
                                         ctypes.byref(io.c), _stream(stream))
    _check(st, "ptd_tree_verify_step_host")
    return last_launch_count()


def draft_tree_update(in_count: torch.Tensor, in_parents: torch.Tensor, in_tokens: torch.Tensor,
                      drafts: torch.Tensor, expand: int, width: int, max_depth: int, capacity: int,
                      out_count: torch.Tensor, out_parents: torch.Tensor, out_tokens: torch.Tensor,
                      out_depths: torch.Tensor, old_to_new: torch.Tensor, dev_status: torch.Tensor, stream=None) -> int:
    """ptd_draft_tree_update.  in_parents / in_tokens / old_to_new: [B, in_stride] int32;
    drafts: [B * in_stride, draft_stride] int32 (a top-k index matrix); out_*: [B, capacity] int32."""
    if in_parents.dim() != 2 or in_tokens.shape != in_parents.shape or old_to_new.shape != in_parents.shape:
        raise ValueError("in_parents, in_tokens and old_to_new must be [batch, in_stride]")
    B, stride = in_parents.shape
    if drafts.dim() != 2 or drafts.shape[0] != B * stride:
        raise ValueError("drafts must be [batch * in_stride, draft_stride]")
    for t, nm in ((out_parents, "out_parents"), (out_tokens, "out_tokens"), (out_depths, "out_depths")):
        if tuple(t.shape) != (B, capacity):
            raise ValueError(f"{nm} must be [batch, capacity]")
    st = lib().ptd_draft_tree_update(
        B, stride, _dev(in_count, "in_count", torch.int32), _dev(in_parents, "in_parents", torch.int32),
        _dev(in_tokens, "in_tokens", torch.int32), _dev(drafts, "drafts", torch.int32), drafts.shape[1],
        int(expand), int(width), int(max_depth), int(capacity), _dev(out_count, "out_count", torch.int32),
        _dev(out_parents, "out_parents", torch.int32), _dev(out_tokens, "out_tokens", torch.int32),
        _dev(out_depths, "out_depths", torch.int32), _dev(old_to_new, "old_to_new", torch.int32),
        _dev(dev_status, "dev_status", torch.int32), _stream(stream))
    _check(st, "ptd_draft_tree_update")
    return last_launch_count()


class CandidatePool:
    """A candidate pool in one device buffer (ptd_pool_bytes / ptd_pool_init)."""

    def __init__(self, capacity: int, device="cuda", stream=None):
        n = int(lib().ptd_pool_bytes(int(capacity)))
        if n == 0:
            raise ValueError("pool capacity must be a power of two in [16, 2^28]")
        self.capacity = int(capacity)
        self.buf = torch.empty(n, dtype=torch.uint8, device=device)
        _check(lib().ptd_pool_init(_dev(self.buf, "pool"), self.capacity, _stream(stream)), "ptd_pool_init")

    def size(self) -> int:
        """Nodes held (reads the device counter: synchronises)."""
        return int(self.buf[:4].view(torch.int32).item())

    def merge(self, step: int, count: torch.Tensor, parents: torch.Tensor, tokens: torch.Tensor,
              dev_status: torch.Tensor, max_load: Optional[int] = None, stream=None) -> int:
        st = lib().ptd_pool_merge(_dev(self.buf, "pool"), self.capacity,
                                  self.capacity // 2 if max_load is None else int(max_load), int(step),
                                  _dev(count, "count", torch.int32), _dev(parents, "parents", torch.int32),
                                  _dev(tokens, "tokens", torch.int32), _dev(dev_status, "dev_status", torch.int32),
                                  _stream(stream))
        _check(st, "ptd_pool_merge")
        return last_launch_count()

    def retrieve(self, root_token: torch.Tensor, width: int, max_depth: int, max_nodes: int,
                 out_count: torch.Tensor, out_parents: torch.Tensor, out_tokens: torch.Tensor, stream=None) -> int:
        if out_parents.numel() < max_nodes or out_tokens.numel() < max_nodes:
            raise ValueError("out_parents / out_tokens need max_nodes entries")
        st = lib().ptd_pool_retrieve(_dev(self.buf, "pool"), self.capacity, _dev(root_token, "root_token", torch.int32),
                                     int(width), int(max_depth), int(max_nodes), _dev(out_count, "out_count", torch.int32),
                                     _dev(out_parents, "out_parents", torch.int32),
                                     _dev(out_tokens, "out_tokens", torch.int32), _stream(stream))
        _check(st, "ptd_pool_retrieve")
        return last_launch_count()


def tree_rope_append(tree: Tree, cache: KVCache, layer_begin: int, q: torch.Tensor, num_q_heads: int,
                     k: torch.Tensor, v: torch.Tensor, rope_base: float, dev_status: torch.Tensor,
                     positions_out: Optional[torch.Tensor] = None, stream=None) -> int:
    """ptd_tree_rope_append: q [L, N_tot, Hq, D] rotated in place; k, v [L, N_tot, Hkv, D]
    into cache layers layer_begin .. layer_begin + L - 1 (a 3-D q, k, v is one layer)."""
    dt = cache.k.dtype
    n_layers = q.shape[0] if q.dim() == 4 else 1
    st = lib().ptd_tree_rope_append(ctypes.byref(tree.c), ctypes.byref(cache.c), int(layer_begin), int(n_layers),
                                    _dev(q, "q", dt),
                                    int(num_q_heads), _dev(k, "k", dt), _dev(v, "v", dt), float(rope_base),
                                    None if positions_out is None else _dev(positions_out, "positions_out", torch.int32),
                                    _dev(dev_status, "dev_status", torch.int32), _stream(stream))
    _check(st, "ptd_tree_rope_append")
    return last_launch_count()


def lm_head_workspace_size(rows: int, vocab: int) -> int:
    return int(lib().ptd_lm_head_topk_workspace_size(int(rows), int(vocab)))


def lm_head_topk(hidden: torch.Tensor, weight: torch.Tensor, k: int, out_idx: torch.Tensor, out_val: torch.Tensor,
                 workspace: torch.Tensor, dev_status: torch.Tensor, stream=None) -> int:
    """ptd_lm_head_topk: hidden [rows, d] and weight [vocab, d] bf16 (rows may be strided)."""
    if hidden.dim() != 2 or weight.dim() != 2 or hidden.shape[1] != weight.shape[1]:
        raise ValueError("hidden [rows, d] and weight [vocab, d] must share d")
    st = lib().ptd_lm_head_topk(_dev(hidden, "hidden", torch.bfloat16, row_strided=True), hidden.shape[0],
                                hidden.stride(0), _dev(weight, "weight", torch.bfloat16, row_strided=True),
                                weight.shape[0], weight.stride(0), hidden.shape[1], int(k),
                                _dev(out_idx, "out_idx", torch.int32), _dev(out_val, "out_val", torch.float32),
                                _dev(workspace, "workspace"), workspace.numel() * workspace.element_size(),
                                _dev(dev_status, "dev_status", torch.int32), _stream(stream))
    _check(st, "ptd_lm_head_topk")
    return last_launch_count()


class Pipeline:
    """ptd_pipeline_*: host-buffer steps with uploads and downloads overlapped with compute.
    trees, bufs: two Tree / StepBuffers sets sharing `cache`; staging: two device byte
    tensors of at least 2 * L * N_tot * Hkv * D elements."""

    def __init__(self, cache: KVCache, trees, bufs, staging, stream=None):
        self.keep = (cache, trees, bufs, staging)
        tr = (_Tree * 2)(trees[0].c, trees[1].c)
        ar = (_StepArgs * 2)(bufs[0].c, bufs[1].c)
        st = (ctypes.c_void_p * 2)(_dev(staging[0], "staging"), _dev(staging[1], "staging"))
        nbytes = min(x.numel() * x.element_size() for x in staging)
        self.h = ctypes.c_void_p()
        _check(lib().ptd_pipeline_create(ctypes.byref(cache.c), tr, ar, st, nbytes, _stream(stream),
                                         ctypes.byref(self.h)), "ptd_pipeline_create")

    def submit(self, io: "HostIO") -> int:
        t = ctypes.c_int64()
        _check(lib().ptd_pipeline_submit(self.h, ctypes.byref(io.c), ctypes.byref(t)), "ptd_pipeline_submit")
        return t.value

    def wait(self, ticket: int) -> None:
        _check(lib().ptd_pipeline_wait(self.h, int(ticket)), "ptd_pipeline_wait")

    def close(self) -> None:
        if self.h:
            lib().ptd_pipeline_destroy(self.h)
            self.h = ctypes.c_void_p()

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass


def check_bounded_wait(dev_status: torch.Tensor, stream=None) -> int:
    """ptd_check_bounded_wait: a wait that runs out, reported as PTD_ERR_TIMEOUT."""
    _check(lib().ptd_check_bounded_wait(_dev(dev_status, "dev_status", torch.int32), _stream(stream)),
           "ptd_check_bounded_wait")
    return last_launch_count()
