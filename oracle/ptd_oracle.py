"""CPU oracle for the Progressive Tree Drafting (PTD) tree-verify step.

TEST INFRASTRUCTURE ONLY.  Nothing on the product path imports this module: only
the tests, `__graft_entry__.smoke()` and the `cpu_baseline` / reference arm of
`bench.py` may call it.  It shares no code with the CUDA kernels.

Plain, slow and written to be checked against the paper by eye.  Floating point
is float64 throughout (bf16 and fp32 inputs are widened exactly).  Every function
cites the passage it follows:

  tree / ancestor sets ......... Sec. 3.1, "Tree Construction": each node sees only
                                 itself and its ancestors, pi(v) = {v} U pi(P(v)).
  tree_attention ............... Sec. 3.1 (ancestor-only visibility) and Sec. 3.2
                                 (one forward pass over [X; T; C_X]): every tree node
                                 attends to the whole committed prefix X plus its own
                                 ancestor set inside the tree.
  topk ......................... Sec. 3.1 "Progressive Expansion" (each node's draft
                                 d_v) and "Width Control" (at most k children);
                                 Sec. 3.2 / Alg. 1 step 5 (greedy V_n = argmax).
  verify_greedy ................ Sec. 3.2, eligible edges I = {(n, V_n) | V_n in
                                 sigma(n)} and the accepted sequence
                                 X' = (n_0, ..., n_k, V_{n_k}); Alg. 1 steps 5-6.
  kv_compact ................... Alg. 1 step 6 (X' is appended to X): the accepted
                                 nodes' K/V become the next committed slots.

Readings where the paper is silent (each listed in the design notes):
  * node 0 of every tree is the current input token (slot C of the cache); draft
    and candidate subtrees hang below it, so one pass is one rooted tree;
  * nodes are in topological order (0 <= parents[i] < i), parents[0] = -1;
  * attention scale 1/sqrt(D); query head h uses KV head h // (Hq/Hkv);
  * top-k ties: the lower vocabulary index first; -0.0 equals +0.0;
  * several eligible children of one node (possible once a draft tree and a
    candidate tree share a root): the longest eligible root path wins, ties broken
    by the lexicographically smallest sequence of node indices;
  * accept_len counts accepted nodes including the root; the bonus token is
    V_{n_k} of the last accepted node.
"""
from __future__ import annotations

import math

import numpy as np


class InvalidTree(ValueError):
    """The parent array does not describe a rooted tree in topological order."""


# ---------------------------------------------------------------------------
# Tree (Sec. 3.1, "Tree Construction")
# ---------------------------------------------------------------------------

def check_tree(parents) -> None:
    """A rooted tree in topological order: parents[0] = -1 and 0 <= parents[i] < i."""
    parents = [int(p) for p in parents]
    if len(parents) == 0 or parents[0] != -1:
        raise InvalidTree("node 0 must be the root (parent -1)")
    for i in range(1, len(parents)):
        if not (0 <= parents[i] < i):
            raise InvalidTree(f"node {i} has parent {parents[i]}")


def ancestor_sets(parents) -> list:
    """pi(v) = {v} U pi(P(v)), with pi(root) = {root}  (Sec. 3.1)."""
    check_tree(parents)
    pi = []
    for v, p in enumerate(int(x) for x in parents):
        pi.append({v} if p < 0 else {v} | pi[p])
    return pi


def depths(parents) -> np.ndarray:
    """Depth of each node = |pi(v)| - 1 (the root has depth 0)."""
    return np.array([len(s) - 1 for s in ancestor_sets(parents)], np.int64)


def children_sets(parents) -> list:
    """sigma(n): the direct children of each node."""
    sig = [[] for _ in parents]
    for c, p in enumerate(int(x) for x in parents):
        if p >= 0:
            sig[p].append(c)
    return sig


# ---------------------------------------------------------------------------
# Tree-masked attention (Sec. 3.1 visibility; Sec. 3.2 combined pass)
# ---------------------------------------------------------------------------

def visibility(parents, ctx_len: int) -> np.ndarray:
    """Boolean [T, C+T]: node i sees every committed slot j < C and the slot C+a of each a in pi(i)."""
    pi = ancestor_sets(parents)
    T = len(pi)
    vis = np.zeros((T, ctx_len + T), dtype=bool)
    vis[:, :ctx_len] = True
    for i, s in enumerate(pi):
        for a in s:
            vis[i, ctx_len + a] = True
    return vis


def tree_attention(q, k, v, parents, ctx_len: int, scale: float | None = None) -> np.ndarray:
    """Tree-masked attention of one sequence in one layer.

    q: [T, Hq, D]; k, v: [>= C+T, Hkv, D], slot j of the sequence in row j (the
    committed prefix in rows [0, C), node i's own K/V in row C+i).  Returns
    o: [T, Hq, D] float64 with, for node i and query head h (KV head h // G),
      s_j = scale * <q[i,h], k[j]>, j visible to i;  p = softmax(s);  o = sum_j p_j v[j].
    """
    q = np.asarray(q, np.float64)
    k = np.asarray(k, np.float64)
    v = np.asarray(v, np.float64)
    T, Hq, D = q.shape
    Hkv = k.shape[1]
    if Hq % Hkv:
        raise ValueError("Hq must be a multiple of Hkv")
    G = Hq // Hkv
    if scale is None:
        scale = 1.0 / math.sqrt(D)
    n = ctx_len + T
    vis = visibility(parents, ctx_len)
    o = np.zeros((T, Hq, D), np.float64)
    for h in range(Hq):
        kv = h // G
        s = scale * (q[:, h, :] @ k[:n, kv, :].T)          # [T, C+T]
        s = np.where(vis, s, -np.inf)
        s = s - s.max(axis=1, keepdims=True)
        p = np.exp(s)
        p = p / p.sum(axis=1, keepdims=True)
        o[:, h, :] = p @ v[:n, kv, :]
    return o


# ---------------------------------------------------------------------------
# Per-node top-k (Sec. 3.1 expansion + width control; greedy V_n)
# ---------------------------------------------------------------------------

def topk(row, k: int):
    """The k largest entries of one logit row: (indices, values), values descending,
    equal values ordered by lower index first (-0.0 equals +0.0).  Entry 0 is the
    row's greedy token (the node's draft d_v and verification token V_n)."""
    x = np.asarray(row, np.float64)
    if not (1 <= k <= x.shape[0]):
        raise ValueError("k out of range")
    order = np.argsort(-x, kind="stable")[:k]     # stable: ties keep index order
    return order.astype(np.int32), x[order]


def topk_rows(logits, k: int):
    """topk applied to each row of a [rows, V] array."""
    x = np.asarray(logits, np.float64)
    idx = np.zeros((x.shape[0], k), np.int32)
    val = np.zeros((x.shape[0], k), np.float64)
    for r in range(x.shape[0]):
        idx[r], val[r] = topk(x[r], k)
    return idx, val


# ---------------------------------------------------------------------------
# Greedy verification (Sec. 3.2, eligible edges I and accepted sequence X')
# ---------------------------------------------------------------------------

def eligible_edges(parents, tokens, target) -> set:
    """I = {(n, c) : c in sigma(n) and token(c) = V_n}, V_n = target[n] (the argmax)."""
    sig = children_sets(parents)
    return {(n, c) for n in range(len(parents)) for c in sig[n] if int(tokens[c]) == int(target[n])}


def verify_greedy(parents, tokens, target):
    """Accepted path X' of one tree: the root path n_0 = 0, n_1, ..., n_k whose edges
    are all in I, the longest such path, ties to the lexicographically smallest node
    sequence.  Returns (path node list, accept_len = k + 1, bonus = V_{n_k})."""
    check_tree(parents)
    I = eligible_edges(parents, tokens, target)
    out = {}
    for (n, c) in sorted(I):
        out.setdefault(n, []).append(c)

    best = [0]

    def walk(path):
        nonlocal best
        if len(path) > len(best) or (len(path) == len(best) and path < best):
            best = list(path)
        for c in out.get(path[-1], []):
            walk(path + [c])

    walk([0])
    return best, len(best), int(target[best[-1]])


# ---------------------------------------------------------------------------
# KV compaction (Alg. 1 step 6: X' joins the committed prefix)
# ---------------------------------------------------------------------------

def kv_compact(cache_seq, path, ctx_len: int):
    """New cache of one sequence: slot C+j takes the (pre-step) content of slot
    C+path[j] for j < len(path); slots below C are untouched; the new committed
    length is C + len(path).  cache_seq: [S, ...] (slot-major).  Returns (new, new_ctx)."""
    snap = np.array(cache_seq, copy=True)
    new = np.array(cache_seq, copy=True)
    for j, n in enumerate(path):
        new[ctx_len + j] = snap[ctx_len + int(n)]
    return new, ctx_len + len(path)
