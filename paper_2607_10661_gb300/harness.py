"""Device-resident buffers of one tree-verify step for a synthetic workload.

Uploads a `synthetic.Workload` (trees, Q, K/V cache, logits, draft tokens) to one GPU and
owns every output buffer, so tests and the benchmark can run the step through the C ABI
(`ptd.tree_verify_step`) or one call at a time.  Layout only: no arithmetic of the step.
"""
from __future__ import annotations

import numpy as np
import torch

from . import ptd
from . import synthetic as syn


def to_torch(a: np.ndarray, dtype: str) -> torch.Tensor:
    """Host numpy array (bf16 bit patterns or fp32) as a torch CPU tensor of the matching dtype."""
    if dtype == "bf16":
        return torch.from_numpy(np.ascontiguousarray(a).view(np.int16)).view(torch.bfloat16)
    return torch.from_numpy(np.ascontiguousarray(a, dtype=np.float32))


class DeviceWorkload:
    def __init__(self, w: syn.Workload, device="cuda:0", with_step_buffers: bool = True):
        self.w = w
        c = w.cfg
        self.device = torch.device(device)
        dev = self.device
        self.tdtype = torch.bfloat16 if c.dtype == "bf16" else torch.float32
        i32 = dict(dtype=torch.int32, device=dev)
        self.node_offsets = torch.tensor(w.node_offsets, **i32)
        self.parents = torch.tensor(w.parents, **i32)
        self.ctx_lens = torch.tensor(w.ctx_lens, **i32)
        self.tree = ptd.Tree(self.node_offsets, self.parents, self.ctx_lens, w.max_nodes, w.max_ctx)
        shape = (c.layers, *w.cache_shape())
        self.k = torch.empty(shape, dtype=self.tdtype, device=dev)
        self.v = torch.empty(shape, dtype=self.tdtype, device=dev)
        self.q = torch.empty((c.layers, w.n_total, c.hq, c.d), dtype=self.tdtype, device=dev)
        for l in range(c.layers):
            kl, vl = w.kv_layer(l)
            self.k[l].copy_(to_torch(kl, c.dtype))
            self.v[l].copy_(to_torch(vl, c.dtype))
            self.q[l].copy_(to_torch(w.q_layer(l), c.dtype))
        self.block_table = torch.tensor(w.block_table, **i32) if c.page_size else None
        self.cache = ptd.KVCache(self.k, self.v, c.hkv, c.d, c.page_size, self.block_table)
        self.logits = to_torch(w.logits, c.dtype).to(dev)
        self.tokens = torch.tensor(w.tokens, **i32)
        self.attn_out = torch.zeros_like(self.q)
        self.topk_idx = torch.zeros((w.n_total, c.k), **i32)
        self.topk_val = torch.zeros((w.n_total, c.k), dtype=torch.float32, device=dev)
        self.accepted = torch.zeros((c.batch, w.max_nodes), **i32)
        self.accept_len = torch.zeros(c.batch, **i32)
        self.bonus = torch.zeros(c.batch, **i32)
        self.new_ctx = torch.zeros(c.batch, **i32)
        self.dev_status = torch.zeros(1, **i32)
        # the step's scratch (the attention's, then the tail's per-tree counters), or the
        # attention's alone for the attention-only workloads
        nbytes = (ptd.step_workspace_size(self.tree, self.cache, c.hq) if with_step_buffers else
                  ptd.attention_workspace_size(self.tree, self.cache, c.hq))
        self.workspace = torch.empty(max(nbytes, 16), dtype=torch.uint8, device=dev) if nbytes else None
        self.bufs = ptd.StepBuffers(self.q, c.hq, self.attn_out, self.logits, c.k, self.tokens, self.topk_idx,
                                    self.topk_val, self.accepted, self.accept_len, self.bonus, self.new_ctx,
                                    self.dev_status, self.workspace) if with_step_buffers else None

    def clone(self) -> "DeviceWorkload":
        """An independent copy of every device buffer (inputs, cache, outputs, workspace) with
        its own Tree / KVCache / StepBuffers descriptions: consecutive benchmark steps can
        alternate between copies so that no step finds the previous one's inputs in L2."""
        new = DeviceWorkload.__new__(DeviceWorkload)
        new.w, new.device, new.tdtype = self.w, self.device, self.tdtype
        c, w = self.w.cfg, self.w
        for name in ("node_offsets", "parents", "ctx_lens", "k", "v", "q", "logits", "tokens", "attn_out", "topk_idx",
                     "topk_val", "accepted", "accept_len", "bonus", "new_ctx", "dev_status"):
            setattr(new, name, getattr(self, name).clone())
        new.block_table = self.block_table.clone() if self.block_table is not None else None
        new.workspace = torch.empty_like(self.workspace) if self.workspace is not None else None
        new.tree = ptd.Tree(new.node_offsets, new.parents, new.ctx_lens, w.max_nodes, w.max_ctx)
        new.cache = ptd.KVCache(new.k, new.v, c.hkv, c.d, c.page_size, new.block_table)
        new.bufs = (ptd.StepBuffers(new.q, c.hq, new.attn_out, new.logits, c.k, new.tokens, new.topk_idx,
                                    new.topk_val, new.accepted, new.accept_len, new.bonus, new.new_ctx,
                                    new.dev_status, new.workspace) if self.bufs is not None else None)
        return new

    # ---- the whole step, or one call at a time ------------------------------------
    def step(self, stream=None) -> int:
        self.dev_status.zero_()
        return ptd.tree_verify_step(self.tree, self.cache, self.bufs, stream)

    def attention(self, stream=None) -> int:
        return ptd.tree_attention(self.tree, self.cache, self.q, self.attn_out, self.w.cfg.hq, self.dev_status,
                                  workspace=self.workspace, stream=stream)

    def topk(self, stream=None) -> int:
        return ptd.topk_draft(self.logits, self.w.cfg.k, self.topk_idx, self.topk_val, stream=stream)

    def verify(self, stream=None) -> int:
        return ptd.verify_greedy(self.tree, self.tokens, self.topk_idx, self.w.cfg.k, self.accepted,
                                 self.accept_len, self.bonus, self.dev_status, stream=stream)

    def verify_and_compact(self, stream=None) -> int:
        return ptd.verify_and_compact(self.tree, self.cache, self.tokens, self.topk_idx, self.w.cfg.k, self.accepted,
                                      self.accept_len, self.bonus, self.new_ctx, self.dev_status, stream=stream)

    def compact(self, stream=None) -> int:
        return ptd.kv_compact(self.tree, self.cache, self.accepted, self.accept_len, self.new_ctx, stream=stream)

    def twin_step_buffers(self):
        """A second (Tree, StepBuffers) set of the same shapes over the same cache: the other
        slot of a two-deep pipeline (ptd.Pipeline).  Nothing is shared with this set."""
        w, c, dev = self.w, self.w.cfg, self.device
        i32 = dict(dtype=torch.int32, device=dev)
        node_offsets, parents, ctx_lens = self.node_offsets.clone(), self.parents.clone(), self.ctx_lens.clone()
        tree = ptd.Tree(node_offsets, parents, ctx_lens, w.max_nodes, w.max_ctx)
        tree.keep = (node_offsets, parents, ctx_lens)
        ws = torch.empty_like(self.workspace) if self.workspace is not None else None
        bufs = ptd.StepBuffers(self.q.clone(), c.hq, torch.zeros_like(self.attn_out), self.logits.clone(), c.k,
                               self.tokens.clone(), torch.zeros_like(self.topk_idx), torch.zeros_like(self.topk_val),
                               torch.zeros_like(self.accepted), torch.zeros((c.batch,), **i32),
                               torch.zeros((c.batch,), **i32), torch.zeros((c.batch,), **i32),
                               torch.zeros(1, **i32), ws)
        return tree, bufs

    def tree_rows(self):
        """The tree's own K and V rows of every layer as they sit in the cache (slots C_b + i),
        [L][N_tot][Hkv][D] each: the `tree_k_h` / `tree_v_h` inputs of a host-buffer step."""
        w = self.w
        outer, inner = [], []
        for b in range(w.cfg.batch):
            o, i = w.slot_rows(b)
            C = int(w.ctx_lens[b])
            outer.append(o[C:])
            inner.append(i[C:])
        o = torch.tensor(np.concatenate(outer), dtype=torch.long, device=self.device)
        i = torch.tensor(np.concatenate(inner), dtype=torch.long, device=self.device)
        return self.k[:, o, i].contiguous(), self.v[:, o, i].contiguous()
