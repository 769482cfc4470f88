"""Seeded synthetic inputs for the Progressive Tree Drafting (PTD) tree-verify step.

This module only draws inputs: random trees, random Q/K/V, random logits and
draft tokens. It computes none of the step's arithmetic (no attention, no top-k,
no verification, no compaction) and it is shared, unchanged, by the CUDA path's
callers (tests, bench) and by the CPU oracle's callers.

Workload shapes follow the paper's setting: batch-size-1 greedy decoding with a
draft tree of max depth 6 and width 4 (Sec. 4.1, Sec. 4.2.2), about 50-75 tree
nodes per step (App. G, drafting/verification tokens), plus a batched paged case
and a long-context case.  No dataset, model or weights exist here: every tensor is
drawn from a counter-seeded numpy PCG64 stream, one stream per (seed, tensor,
layer), so any single layer can be regenerated on its own.

Recipe (all configs):
  * Q, K, V ~ N(0, 1) in fp32, rounded to bf16 with round-to-nearest-even for the
    bf16 configs.  The cache holds the committed context (slots [0, C)) followed by
    the tree nodes' own K/V (slot C + i for node i), Sec. 3.2 ([X; T; C_X] in one
    pass).
  * Trees are parent-pointer arrays in BFS order, parents[0] = -1.  A "branching"
    tree is the full tree of the branching list, pruned to T nodes by keeping one
    random full-depth spine and then repeatedly adding the highest random score
    node among the children of kept nodes.
  * Logits ~ N(0, sigma) with one planted target token per node raised by +boost.
  * Draft tokens: for each child (in order) of node p, with probability p_match,
    and only if no earlier sibling matched, the child's token is the row argmax of
    p's logits (numpy's first-occurrence argmax on the rounded values, used only to
    shape acceptance statistics); otherwise a uniform token that differs from that
    argmax and from earlier siblings' tokens.  The root token is uniform.
"""
from __future__ import annotations

import dataclasses
from typing import Optional

import numpy as np

# Stream ids for the per-tensor generators.
_S_TREE, _S_LOGITS, _S_TOKENS, _S_Q, _S_K, _S_V, _S_PAGES, _S_CTX = range(8)


def rng(seed: int, *stream: int) -> np.random.Generator:
    """Counter-style seeding: one independent PCG64 stream per (seed, stream...)."""
    return np.random.Generator(np.random.PCG64(np.random.SeedSequence([int(seed), *map(int, stream)])))


def bf16_bits(x: np.ndarray) -> np.ndarray:
    """Round fp32 values to bf16 (round to nearest, ties to even); returns uint16 bit patterns.
    Inputs are finite (the generator draws no NaN/Inf)."""
    u = np.ascontiguousarray(x, dtype=np.float32).view(np.uint32)
    r = u + np.uint32(0x7FFF) + ((u >> np.uint32(16)) & np.uint32(1))
    return (r >> np.uint32(16)).astype(np.uint16)


def bf16_to_f32(bits: np.ndarray) -> np.ndarray:
    """Exact widening of bf16 bit patterns to fp32."""
    return (np.ascontiguousarray(bits, dtype=np.uint16).astype(np.uint32) << np.uint32(16)).view(np.float32)


# --------------------------------------------------------------------------------------
# Workload configurations
# --------------------------------------------------------------------------------------

@dataclasses.dataclass(frozen=True)
class Config:
    name: str
    dtype: str                 # "f32" or "bf16"
    batch: int
    layers: int
    hq: int
    hkv: int
    d: int
    vocab: int
    k: int
    sigma: float
    boost: float
    p_match: float
    ctx: tuple                 # (lo, hi) inclusive; lo == hi for a fixed context
    tree: str                  # "binary" | "branching" | "random-depth"
    nodes: tuple               # (lo, hi) node count range
    branching: tuple = ()
    depth_range: tuple = ()
    page_size: int = 0         # 0 = contiguous cache


CONFIGS = {
    # Tiny fp32 single layer: complete binary tree of 15 nodes (4 levels), 8 MHA heads, D 64.
    "tiny-fp32": Config("tiny-fp32", "f32", 1, 1, 8, 8, 64, 1000, 2, 1.0, 4.0, 0.6,
                        (256, 256), "binary", (15, 15)),
    # Llama-2-7B-shaped layer: 32 MHA heads, context 2048, branching (3,2,2,1,1) pruned to 31.
    "llama2-7b-layer": Config("llama2-7b-layer", "bf16", 1, 1, 32, 32, 128, 32000, 3, 2.0, 5.0, 0.5,
                              (2048, 2048), "branching", (31, 31), branching=(3, 2, 2, 1, 1)),
    # Llama-3-8B-shaped GQA stack: 32 layers, 32q/8kv, context 8192, branching (4,3,2,2,1,1) -> 63.
    "llama3-8b-gqa": Config("llama3-8b-gqa", "bf16", 1, 32, 32, 8, 128, 128256, 4, 2.0, 6.0, 0.55,
                            (8192, 8192), "branching", (63, 63), branching=(4, 3, 2, 2, 1, 1)),
    # Batched serving: 8 sequences, ragged contexts in [1024, 4096], 16-token pages.
    "batched-paged": Config("batched-paged", "bf16", 8, 1, 32, 8, 128, 128256, 4, 2.0, 6.0, 0.5,
                            (1024, 4096), "random-depth", (16, 64), branching=(4, 3, 2, 2, 1, 1, 1),
                            depth_range=(3, 7), page_size=16),
    # Long context: 64q/8kv, context 32768, branching (6,4,2,2,1,1,1,1) -> 128.
    "long-context": Config("long-context", "bf16", 1, 1, 64, 8, 128, 152064, 6, 2.0, 6.0, 0.45,
                           (32768, 32768), "branching", (128, 128), branching=(6, 4, 2, 2, 1, 1, 1, 1)),
}

CONFIG_ORDER = ["tiny-fp32", "llama2-7b-layer", "llama3-8b-gqa", "batched-paged", "long-context"]


def shrink(cfg: Config, **changes) -> Config:
    """A copy of `cfg` with some fields replaced (smaller parity cases of the same shape)."""
    return dataclasses.replace(cfg, **changes)


# --------------------------------------------------------------------------------------
# Trees
# --------------------------------------------------------------------------------------

def full_tree(branching) -> tuple[np.ndarray, np.ndarray]:
    """Full tree of a branching list in BFS order: parents and levels."""
    parents, levels = [-1], [0]
    frontier = [0]
    for lvl, b in enumerate(branching, start=1):
        nxt = []
        for p in frontier:
            for _ in range(b):
                parents.append(p)
                levels.append(lvl)
                nxt.append(len(parents) - 1)
        frontier = nxt
    return np.array(parents, np.int64), np.array(levels, np.int64)


def _bfs_relabel(parents: np.ndarray, keep: np.ndarray) -> np.ndarray:
    """Relabel the kept nodes of a tree (given in BFS order) in BFS order."""
    kept = sorted(int(i) for i in keep)           # original BFS order is preserved
    new_id = {old: new for new, old in enumerate(kept)}
    out = np.empty(len(kept), np.int32)
    for old in kept:
        p = int(parents[old])
        out[new_id[old]] = -1 if p < 0 else new_id[p]
    return out


def pruned_tree(branching, n_nodes: int, g: np.random.Generator) -> np.ndarray:
    """Full tree of `branching`, pruned to `n_nodes` nodes by random scores; BFS order."""
    parents, levels = full_tree(branching)
    n_full = len(parents)
    n_nodes = min(n_nodes, n_full)
    children = [[] for _ in range(n_full)]
    for c in range(1, n_full):
        children[parents[c]].append(c)
    score = g.random(n_full)
    keep = set()
    # one random root-to-leaf spine of full depth
    v = 0
    keep.add(0)
    while children[v]:
        v = children[v][int(g.integers(len(children[v])))]
        keep.add(v)
    if len(keep) > n_nodes:             # the spine alone is deeper than the budget
        spine = sorted(keep)[:n_nodes]
        keep = set(spine)
    while len(keep) < n_nodes:
        frontier = [c for v in keep for c in children[v] if c not in keep]
        best = max(frontier, key=lambda c: (score[c], -c))
        keep.add(best)
    return _bfs_relabel(parents, np.array(sorted(keep)))


def binary_tree(n_nodes: int) -> np.ndarray:
    """Complete binary tree in BFS order: parent of i is (i-1)//2."""
    p = np.array([(i - 1) // 2 for i in range(n_nodes)], np.int32)
    p[0] = -1
    return p


# --------------------------------------------------------------------------------------
# Workload
# --------------------------------------------------------------------------------------

class Workload:
    """All inputs of one tree-verify step for a config and a seed.

    Small tensors (trees, tokens, logits) are materialised on construction; the
    per-layer Q/K/V are drawn on demand so one layer can be regenerated alone.

    Layouts (host numpy arrays):
      parents      int32 [N_tot]   tree-local parent of each node, trees back to back
      node_offsets int32 [B+1]
      ctx_lens     int32 [B]       committed context C_b; node i of tree b at slot C_b + i
      tokens       int32 [N_tot]   draft token of each node
      logits       [N_tot, V]      uint16 bf16 bits or float32
      q_layer(l)   [N_tot, Hq, D]
      kv_layer(l)  (K, V), each [B, S_cap, Hkv, D] (contiguous) or [P, page, Hkv, D] (paged)
      block_table  int32 [B, max_pages] (paged only)
    """

    def __init__(self, cfg: Config, seed: int):
        self.cfg = cfg
        self.seed = int(seed)
        B = cfg.batch
        gt = rng(seed, _S_TREE)
        trees = []
        for b in range(B):
            if cfg.tree == "binary":
                trees.append(binary_tree(cfg.nodes[0]))
            elif cfg.tree == "branching":
                trees.append(pruned_tree(cfg.branching, cfg.nodes[0], gt))
            elif cfg.tree == "random-depth":
                depth = int(gt.integers(cfg.depth_range[0], cfg.depth_range[1] + 1))
                t = int(gt.integers(cfg.nodes[0], cfg.nodes[1] + 1))
                trees.append(pruned_tree(cfg.branching[:depth], t, gt))
            elif cfg.tree == "chain":
                t = cfg.nodes[0]
                trees.append(np.arange(-1, t - 1, dtype=np.int32))
            else:
                raise ValueError(cfg.tree)
        self.trees = trees
        self.parents = np.concatenate(trees).astype(np.int32)
        self.node_offsets = np.zeros(B + 1, np.int32)
        self.node_offsets[1:] = np.cumsum([len(t) for t in trees])
        self.n_total = int(self.node_offsets[-1])
        self.max_nodes = max(len(t) for t in trees)
        gc = rng(seed, _S_CTX)
        self.ctx_lens = gc.integers(cfg.ctx[0], cfg.ctx[1] + 1, size=B).astype(np.int32)
        self.seq_lens = self.ctx_lens + np.array([len(t) for t in trees], np.int32)
        self.max_ctx = int(self.ctx_lens.max())

        # logits and planted targets
        gl = rng(seed, _S_LOGITS)
        V = cfg.vocab
        raw = gl.standard_normal((self.n_total, V), dtype=np.float32) * np.float32(cfg.sigma)
        planted = gl.integers(0, V, size=self.n_total)
        raw[np.arange(self.n_total), planted] += np.float32(cfg.boost)
        if cfg.dtype == "bf16":
            self.logits = bf16_bits(raw)
            widened = bf16_to_f32(self.logits)
        else:
            self.logits = raw
            widened = raw
        self.planted = planted.astype(np.int32)
        # input shaping only: which token a matching draft child carries
        row_argmax = np.argmax(widened, axis=1)

        # draft tokens
        gk = rng(seed, _S_TOKENS)
        tokens = np.empty(self.n_total, np.int32)
        for b, par in enumerate(trees):
            off = int(self.node_offsets[b])
            tokens[off] = int(gk.integers(V))
            kids = [[] for _ in range(len(par))]
            for c in range(1, len(par)):
                kids[par[c]].append(c)
            for p, ch in enumerate(kids):
                target = int(row_argmax[off + p])
                used = set()
                matched = False
                for c in ch:
                    if not matched and gk.random() < cfg.p_match:
                        tok = target
                        matched = True
                    else:
                        while True:
                            tok = int(gk.integers(V))
                            if tok != target and tok not in used:
                                break
                    used.add(tok)
                    tokens[off + c] = tok
        self.tokens = tokens

        # cache geometry
        if cfg.page_size:
            ps = cfg.page_size
            pages_per_seq = [(int(s) + ps - 1) // ps for s in self.seq_lens]
            self.max_pages = max(pages_per_seq)
            self.num_pages = int(sum(pages_per_seq)) + 3          # a few spare pages
            perm = rng(seed, _S_PAGES).permutation(self.num_pages).astype(np.int32)
            self.block_table = np.full((B, self.max_pages), -1, np.int32)
            at = 0
            for b, n in enumerate(pages_per_seq):
                self.block_table[b, :n] = perm[at:at + n]
                at += n
            self.seq_capacity = 0
        else:
            self.block_table = None
            self.max_pages = 0
            self.num_pages = 0
            self.seq_capacity = int(self.seq_lens.max())

    # ---- per-layer tensors --------------------------------------------------------
    def _draw(self, stream: int, layer: int, shape):
        x = rng(self.seed, stream, layer).standard_normal(shape, dtype=np.float32)
        return bf16_bits(x) if self.cfg.dtype == "bf16" else x

    def cache_shape(self):
        c = self.cfg
        if c.page_size:
            return (self.num_pages, c.page_size, c.hkv, c.d)
        return (c.batch, self.seq_capacity, c.hkv, c.d)

    def q_layer(self, layer: int) -> np.ndarray:
        c = self.cfg
        return self._draw(_S_Q, layer, (self.n_total, c.hq, c.d))

    def kv_layer(self, layer: int):
        shape = self.cache_shape()
        return self._draw(_S_K, layer, shape), self._draw(_S_V, layer, shape)

    # ---- logical views (layout only) ---------------------------------------------
    def slot_rows(self, b: int, n_slots: Optional[int] = None) -> tuple:
        """Physical (outer, inner) row indices of sequence b's first n_slots cache slots."""
        n = int(self.seq_lens[b]) if n_slots is None else int(n_slots)
        s = np.arange(n)
        if self.cfg.page_size:
            ps = self.cfg.page_size
            return self.block_table[b, s // ps], s % ps
        return np.full(n, b), s

    def seq_view(self, cache_layer: np.ndarray, b: int, n_slots: Optional[int] = None) -> np.ndarray:
        """Sequence b's slots [0, n) of one layer's cache tensor as [n, Hkv, D]."""
        o, i = self.slot_rows(b, n_slots)
        return cache_layer[o, i]

    def tree(self, b: int) -> np.ndarray:
        return self.trees[b]

    def nodes_of(self, b: int) -> slice:
        return slice(int(self.node_offsets[b]), int(self.node_offsets[b + 1]))


def widen(x: np.ndarray, dtype: str) -> np.ndarray:
    """Exact float64 view of generator values (bf16 bits or fp32)."""
    if dtype == "bf16":
        return bf16_to_f32(x).astype(np.float64)
    return np.asarray(x, np.float32).astype(np.float64)
