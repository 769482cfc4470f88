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
  verify_sampling .............. Sec. 3.2, "sampling decoding strategy", and Alg. 2
                                 (Candidate Tree Recursive Sampling), whose output
                                 distribution App. E proves to be P.
  draft_tree_update ............ Sec. 3.1 "Progressive Expansion" (every node's draft
                                 token joins the tree as its child), "Width Control"
                                 and "Stepping Mechanism (Depth Control)"; Alg. 1
                                 step 3 (expand, then StepAndPrune past d_max).
  lm_head_topk ................. the per-node logits P(y_T | ...) of Alg. 1 step 2 as
                                 the LM-head product h_v W^T, followed by topk_rows
                                 (the drafts d_v and verification tokens V_n).
  tree_positions, rope ......... Sec. 3.1 "Tree Construction": a node's position is
                                 set by |pi(v)|, here C + |pi(v)| - 1 after the
                                 committed prefix; the rotary encoding itself is the
                                 model's (RoFormer's rotation, rotate-half layout).
  CandidatePool ................ Sec. 3.1 "Draft Extraction via Merging" (the merge
                                 M(T, T') of two trees with the same root value) and
                                 Alg. 1 step 4; Sec. 3.2 and Alg. 1 step 1 (retrieve
                                 the candidate tree C_X for the decoded sequence X).

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
  * sampling verification: P_v = softmax(logits_v / temperature); each child of the
    current node is tried once, in node order, with its own uniform r: accepted when
    r < P(token)/S, S being the mass of P_v not yet rejected (Alg. 2 writes "<", the
    text of Sec. 3.2 "<=": they differ on a set of measure zero); a rejected token's
    probability becomes 0 (a later sibling with the same token then has probability
    0).  Alg. 2 wraps this in "while C is not empty", which as printed never ends when
    every child is rejected; App. E and Sec. 3.2 try each candidate once, as here.
    With no child accepted (or at a leaf) the bonus token is drawn from the residual
    P_v / S by inverse CDF in vocabulary order with the tree's own uniform.  The
    uniforms are inputs, so the kernel and this oracle see the same random numbers.
  * draft tree update: the draft tree is a forest of seed subtrees (a seed's parent
    is -1; in a verification pass they hang below node 0) stored in creation order,
    so a parent precedes its children and "earliest added" means "lowest index".
    Expansion visits the nodes in index order and each node's draft tokens in rank
    order (the first `expand` of its top-k row); a token equal to an existing
    child's is that child (V is a set of (parent, token) nodes), not a new node;
    width control caps a node's children at `width`; new nodes are appended in that
    visiting order while the forest has fewer than `capacity` nodes.  Depth control
    applies per seed subtree ("when a sub-tree exceeds a depth threshold"): depth
    counts nodes on the longest seed-to-leaf path (a lone seed has depth 1); a
    subtree deeper than d_max is replaced by the subtree of the seed's lowest-index
    child, which becomes a seed; everything else under the old seed goes.  Pruning
    runs once per step, after expansion (Alg. 1 step 3).  Survivors keep their
    relative order.
  * tree positions: node v of a tree over a committed prefix of C tokens sits at
    position C + |pi(v)| - 1 (the root, the current input token, at C: the position
    the next token of plain decoding would have); the rotary encoding is RoFormer's
    rotation in the rotate-half layout used by Llama-family models: dims i and i + D/2
    turn by pos * base^(-2i/D).
  * candidate pool: a map from a root token to a trie of draft continuations.  The
    merge M is read as the union of tries: a child of T' whose token is not among the
    children of T joins T together with its whole subtree (the printed case adds the
    child node; its subtree follows by applying the same rule below it), and a child
    whose token is there is merged recursively.  "Any subtree T' of T^t" is every
    node's subtree: after each step, for every node v of the draft forest in index
    order, the subtree rooted at v is merged into the pool entry of token(v) (created
    when absent).  Children keep their order of insertion.  Retrieval for the decoded
    sequence X takes the entry of X's last token (the current input token, node 0 of
    the verification pass) and lays it out breadth first: at most `width` children per
    node, the earliest inserted first, nodes of depth at most `max_depth` (the root
    has depth 1), at most `max_nodes` nodes in that order.  A token with no entry
    gives the lone root.
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
# Sampling verification (Sec. 3.2 "sampling decoding strategy"; Alg. 2; App. E)
# ---------------------------------------------------------------------------

def softmax_row(logits_row, temperature: float = 1.0) -> np.ndarray:
    """P_v: the target model's distribution over the next token at node v (Sec. 3.2),
    softmax of the node's logits divided by the temperature, in float64."""
    x = np.asarray(logits_row, dtype=np.float64) / float(temperature)
    e = np.exp(x - x.max())
    return e / e.sum()


def verify_sampling(parents, tokens, logits, temperature, u_accept, u_bonus):
    """Sampling verification of one tree (Alg. 2, Candidate Tree Recursive Sampling).

    From the root, the children sigma(v) of the current node v are tried in node order;
    child n is accepted when u_accept[n] < P_v[tokens[n]] / S, where S is the mass of P_v
    not yet rejected; a rejected child's token gets probability 0 (P renormalised over
    the rest).  An accepted child becomes the current node.  When no child is accepted
    (or v is a leaf) the bonus token is drawn from the residual P_v / S by inverse CDF
    with u_bonus.  logits: [T, V] rows of this tree.  Returns (path, accept_len, bonus,
    margin) where margin is the smallest distance between a uniform and the threshold it
    was compared with (acceptance tests and the bonus CDF), a measure of how far every
    decision is from flipping."""
    check_tree(parents)
    sigma = children_sets(parents)
    path = [0]
    v = 0
    margin = math.inf
    while True:
        P = softmax_row(logits[v], temperature)
        S = 1.0
        chosen = None
        for n in sigma[v]:
            t = int(tokens[n])
            p_hat = P[t] / S if S > 0.0 else 0.0
            r = float(u_accept[n])
            margin = min(margin, abs(r - p_hat))
            if r < p_hat:
                chosen = n
                break
            S -= P[t]
            P[t] = 0.0
        if chosen is None:
            break
        path.append(chosen)
        v = chosen
    # no child selected: a sample from the residual distribution of the current node
    target = float(u_bonus) * S
    cdf = np.cumsum(P)
    above = np.nonzero(cdf > target)[0]
    bonus = int(above[0]) if len(above) else int(np.nonzero(P > 0.0)[0][-1])
    lo = cdf[bonus - 1] if bonus > 0 else 0.0
    margin = min(margin, abs(target - lo) / max(S, 1e-300), abs(cdf[bonus] - target) / max(S, 1e-300))
    return path, len(path), bonus, margin


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


# ---------------------------------------------------------------------------
# Draft tree update (Sec. 3.1 "Progressive Expansion", "Width Control",
# "Stepping Mechanism"; Alg. 1 step 3)
# ---------------------------------------------------------------------------

def check_forest(parents) -> None:
    """A forest in creation order: parents[i] = -1 (a seed) or 0 <= parents[i] < i."""
    for i, p in enumerate(parents):
        if not (p == -1 or 0 <= int(p) < i):
            raise InvalidTree(f"node {i}: parent {p} is neither -1 nor an earlier node")


def draft_tree_update(parents, tokens, drafts, expand: int, width: int, max_depth: int, capacity: int):
    """One step of the draft forest's evolution: T^{t-1} -> T^t.

    parents, tokens: the forest T^{t-1} (seeds have parent -1), creation order.
    drafts[v]: node v's draft tokens in rank order (its top-k row); the first
    `expand` are appended as children of v (Sec. 3.1: V^t = V^{t-1} U {d_v},
    E^t = E^{t-1} U {(v, d_v)}), subject to width control (at most `width` children
    per node) and to `capacity` nodes in all.  Then every seed subtree deeper than
    `max_depth` is stepped (Alg. 1 StepAndPrune): its seed's earliest-added child
    becomes the seed of what is kept, the rest of the subtree is pruned.

    Returns (new_parents, new_tokens, new_depths, old_to_new) where new_depths[i] =
    |pi(i)| in the new forest (the node's position offset, Sec. 3.1) and
    old_to_new[j] is the new index of input node j, or -1 if it was pruned."""
    check_forest(parents)
    T = len(parents)
    if T > capacity:
        raise ValueError("the input forest is larger than the capacity")
    par = [int(p) for p in parents]
    tok = [int(t) for t in tokens]
    origin = list(range(T))            # input index of each node, -1 for a new node

    # ---- Step 3, expansion: every node appends its draft tokens as children
    for v in range(T):
        for r in range(expand):
            d = int(drafts[v][r])
            kids = [i for i in range(len(par)) if par[i] == v]
            if any(tok[i] == d for i in kids):
                continue                 # (v, d) is already in V
            if len(kids) >= width or len(par) >= capacity:
                continue                 # width control / no room
            par.append(v)
            tok.append(d)
            origin.append(-1)

    # ---- depth of every node: |pi(v)|
    n = len(par)
    depth = [0] * n
    seed = [0] * n
    for i in range(n):
        depth[i] = 1 if par[i] == -1 else depth[par[i]] + 1
        seed[i] = i if par[i] == -1 else seed[par[i]]

    # ---- StepAndPrune: per seed subtree deeper than max_depth
    keep = [True] * n
    new_seed = {}
    for s in range(n):
        if par[s] != -1:
            continue
        sub_depth = max(depth[i] for i in range(n) if seed[i] == s)
        if sub_depth <= max_depth:
            continue
        first_child = min(i for i in range(n) if par[i] == s)   # earliest added
        new_seed[s] = first_child
        for i in range(n):
            if seed[i] != s:
                continue
            a = i                        # is first_child an ancestor of i (or i itself)?
            while a != -1 and a != first_child:
                a = par[a]
            keep[i] = a == first_child

    # ---- survivors, in order
    new_index = [-1] * n
    m = 0
    for i in range(n):
        if keep[i]:
            new_index[i] = m
            m += 1
    new_par, new_tok, new_dep = [], [], []
    for i in range(n):
        if not keep[i]:
            continue
        p = par[i]
        new_par.append(-1 if (p == -1 or not keep[p]) else new_index[p])
        new_tok.append(tok[i])
    for i in range(m):
        new_dep.append(1 if new_par[i] == -1 else new_dep[new_par[i]] + 1)
    old_to_new = [new_index[j] for j in range(T)]
    return (np.array(new_par, np.int64), np.array(new_tok, np.int64), np.array(new_dep, np.int64),
            np.array(old_to_new, np.int64))


# ---------------------------------------------------------------------------
# Candidate pool (Sec. 3.1 "Draft Extraction via Merging"; Sec. 3.2; Alg. 1 steps 1, 4)
# ---------------------------------------------------------------------------

class _PoolNode:
    __slots__ = ("token", "children")

    def __init__(self, token: int):
        self.token = token
        self.children = []            # insertion order


class CandidatePool:
    """Root token -> trie of draft continuations."""

    def __init__(self):
        self.roots = {}

    def size(self) -> int:
        """Nodes held (roots included)."""
        def count(n):
            return 1 + sum(count(c) for c in n.children)
        return sum(count(r) for r in self.roots.values())

    def _merge(self, pnode, parents, tokens, kids, v):
        """M(P, T'_v): merge the children of draft node v under pool node pnode."""
        for c in kids[v]:
            tok = int(tokens[c])
            match = next((x for x in pnode.children if x.token == tok), None)
            if match is None:                  # sigma(T') \ sigma(T): joins with its subtree
                match = _PoolNode(tok)
                pnode.children.append(match)
            self._merge(match, parents, tokens, kids, c)   # sigma(T') n sigma(T): recurse

    def merge_forest(self, parents, tokens) -> None:
        """Alg. 1 step 4: every node's subtree of the draft forest T^t joins the pool
        entry of its root token, nodes in index order."""
        check_forest(parents)
        kids = [[] for _ in parents]
        for i, p in enumerate(parents):
            if p >= 0:
                kids[p].append(i)
        for v in range(len(parents)):
            tok = int(tokens[v])
            if tok not in self.roots:
                self.roots[tok] = _PoolNode(tok)
            self._merge(self.roots[tok], parents, tokens, kids, v)

    def retrieve(self, root_token: int, width: int, max_depth: int, max_nodes: int):
        """Alg. 1 step 1: the candidate tree C_X for a sequence whose last token is
        root_token, breadth first (parents, tokens), node 0 the root."""
        root = self.roots.get(int(root_token))
        parents, tokens = [-1], [int(root_token)]
        if root is None:
            return np.array(parents, np.int64), np.array(tokens, np.int64)
        frontier = [(root, 0)]                 # (pool node, its index in the output)
        depth = 1
        while frontier and depth < max_depth and len(tokens) < max_nodes:
            nxt = []
            for node, idx in frontier:
                for c in node.children[:width]:
                    if len(tokens) >= max_nodes:
                        break
                    parents.append(idx)
                    tokens.append(c.token)
                    nxt.append((c, len(tokens) - 1))
            frontier = nxt
            depth += 1
        return np.array(parents, np.int64), np.array(tokens, np.int64)


# ---------------------------------------------------------------------------
# Tree positions and the rotary encoding (Sec. 3.1 "Tree Construction")
# ---------------------------------------------------------------------------

def tree_positions(parents, ctx_len: int) -> np.ndarray:
    """Position of every node: C + |pi(v)| - 1 (|pi(v)| counts v and its ancestors)."""
    return np.asarray([ctx_len + len(a) - 1 for a in ancestor_sets(parents)], np.int64)


def rope(x, positions, base: float) -> np.ndarray:
    """Rotary encoding of x [N, H, D] at positions [N] (float64): for i < D/2 the pair
    (x_i, x_{i+D/2}) turns by the angle positions[n] * base^(-2i/D)."""
    x = np.asarray(x, np.float64)
    D = x.shape[-1]
    half = D // 2
    inv_freq = base ** (-2.0 * np.arange(half, dtype=np.float64) / D)
    ang = np.asarray(positions, np.float64)[:, None] * inv_freq[None, :]        # [N, D/2]
    c, s = np.cos(ang)[:, None, :], np.sin(ang)[:, None, :]
    a, b = x[..., :half], x[..., half:]
    return np.concatenate([a * c - b * s, a * s + b * c], axis=-1)


# ---------------------------------------------------------------------------
# LM head with top-k (Alg. 1 step 2: the per-node logits; Sec. 3.1 / 3.2: their top-k)
# ---------------------------------------------------------------------------

def lm_head_logits(hidden, weight) -> np.ndarray:
    """Logits of every node: hidden [N, d] times weight [V, d] transposed, in float64."""
    return np.asarray(hidden, np.float64) @ np.asarray(weight, np.float64).T


def lm_head_topk(hidden, weight, k: int):
    """topk_rows of the LM-head logits: (indices [N, k], values [N, k])."""
    return topk_rows(lm_head_logits(hidden, weight), k)
