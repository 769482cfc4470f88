"""Pins of the CPU oracle against things other than itself (no GPU needed).

Each check is chosen so that a plausible slip in the oracle (a dropped ancestor, a
wrong GQA head map, a missing context slot, a reversed tie-break, a transposed
operand, an unsafe overlapping copy) fails at least one of them:
  * hand-derived worked examples (tests/golden/*.json, each citing its passage);
  * reductions to library routines: float64 torch SDPA with masks built without
    the ancestor sets (chain = causal chunk, single node = plain decode, star),
    np.lexsort for top-k;
  * closed forms (identical keys -> mean of the visible values);
  * brute force: every root path of every recursive tree with <= 7 nodes under
    every binary token/target assignment;
  * invariants and metamorphic relabelling.
"""
import itertools
import json
import math
import os
from fractions import Fraction

import numpy as np
import pytest
import torch

import oracle
from paper_2607_10661_gb300 import synthetic as syn

GOLD = os.path.join(os.path.dirname(__file__), "golden")


def _load(name):
    with open(os.path.join(GOLD, name)) as f:
        return json.load(f)


def _num(x):
    if isinstance(x, (int, float)):
        return float(x)
    if x.startswith("ln"):
        return math.log(float(x[2:]))
    return float(Fraction(x))


# ----------------------------------------------------------------------------- tree

def test_check_tree_rejects_bad_parents():
    for bad in ([], [0], [-1, 1], [-1, 0, 2], [-1, -1], [-1, 0, 5], [1, -1]):
        with pytest.raises(oracle.InvalidTree):
            oracle.check_tree(bad)
    oracle.check_tree([-1])
    oracle.check_tree([-1, 0, 0, 1, 3])


def test_ancestor_sets_closed_forms():
    # chain: pi(i) = {0..i};  complete binary: |pi(i)| = floor(log2(i+1)) + 1
    chain = [-1] + list(range(0, 9))
    for i, s in enumerate(oracle.ancestor_sets(chain)):
        assert s == set(range(i + 1))
    b = syn.binary_tree(31)
    for i, s in enumerate(oracle.ancestor_sets(b)):
        assert len(s) == int(math.floor(math.log2(i + 1))) + 1
        # every member's own ancestors are a subset (closure)
        assert all(((j - 1) // 2 in s) for j in s if j > 0)


# ------------------------------------------------------------------------ attention

def test_attention_worked_example():
    g = _load("attention_worked.json")
    C, scale, parents = g["ctx_len"], g["scale"], g["parents"]
    q = np.stack([np.array(g["q_head0"], float), np.array(g["q_head1"], float)], axis=1)  # [T,2,D]
    k = np.array([[_num(x) for x in r] for r in g["k"]])[:, None, :]
    v = np.array([[_num(x) for x in r] for r in g["v"]])[:, None, :]
    o = oracle.tree_attention(q, k, v, parents, C, scale)
    exp0 = np.array([[_num(x) for x in r] for r in g["o_head0"]])
    exp1 = np.array([[_num(x) for x in r] for r in g["o_head1"]])
    np.testing.assert_allclose(o[:, 0, :], exp0, rtol=0, atol=1e-13)
    np.testing.assert_allclose(o[:, 1, :], exp1, rtol=0, atol=1e-13)


def _sdpa(q, k, v, mask, scale):
    """float64 torch SDPA: q [T,H,D], k/v [N,H,D], mask [T,N] bool (True = attend)."""
    qt = torch.from_numpy(q).permute(1, 0, 2)[None]
    kt = torch.from_numpy(k).permute(1, 0, 2)[None]
    vt = torch.from_numpy(v).permute(1, 0, 2)[None]
    o = torch.nn.functional.scaled_dot_product_attention(
        qt, kt, vt, attn_mask=torch.from_numpy(mask), scale=scale)
    return o[0].permute(1, 0, 2).numpy()


def _rand_qkv(seed, T, C, Hq, Hkv, D):
    g = np.random.default_rng(seed)
    return (g.standard_normal((T, Hq, D)), g.standard_normal((C + T, Hkv, D)),
            g.standard_normal((C + T, Hkv, D)))


@pytest.mark.parametrize("C", [0, 1, 7, 40])
def test_chain_tree_is_causal_chunk(C):
    T, H, D = 9, 3, 16
    q, k, v = _rand_qkv(1 + C, T, C, H, H, D)
    parents = [-1] + list(range(T - 1))
    mask = np.tril(np.ones((T, C + T), bool), k=C)       # causal over an appended chunk
    o = oracle.tree_attention(q, k, v, parents, C)
    np.testing.assert_allclose(o, _sdpa(q, k, v, mask, 1 / math.sqrt(D)), rtol=1e-12, atol=1e-12)


@pytest.mark.parametrize("C", [0, 5, 300])
def test_single_node_is_plain_decode(C):
    H, D = 4, 32
    q, k, v = _rand_qkv(7 + C, 1, C, H, H, D)
    o = oracle.tree_attention(q, k, v, [-1], C)
    mask = np.ones((1, C + 1), bool)
    np.testing.assert_allclose(o, _sdpa(q, k, v, mask, 1 / math.sqrt(D)), rtol=1e-12, atol=1e-12)


def test_star_tree_sees_context_root_self():
    T, C, H, D = 6, 11, 2, 8
    q, k, v = _rand_qkv(3, T, C, H, H, D)
    parents = [-1] + [0] * (T - 1)
    mask = np.zeros((T, C + T), bool)
    mask[:, :C + 1] = True                               # context and the root
    mask[np.arange(T), C + np.arange(T)] = True          # itself
    o = oracle.tree_attention(q, k, v, parents, C)
    np.testing.assert_allclose(o, _sdpa(q, k, v, mask, 1 / math.sqrt(D)), rtol=1e-12, atol=1e-12)


@pytest.mark.parametrize("G", [1, 4, 8])
def test_gqa_matches_repeated_kv_heads(G):
    """Query head h uses KV head h // G: equals MHA with each KV head repeated G times.
    The mask is the complete binary tree's, built from (i-1)//2 without ancestor sets."""
    T, C, Hkv, D = 15, 20, 2, 16
    q, k, v = _rand_qkv(11 * G, T, C, Hkv * G, Hkv, D)
    parents = syn.binary_tree(T)
    mask = np.zeros((T, C + T), bool)
    mask[:, :C] = True
    for i in range(T):
        a = i
        while True:
            mask[i, C + a] = True
            if a == 0:
                break
            a = (a - 1) // 2
    o = oracle.tree_attention(q, k, v, parents, C)
    kr, vr = np.repeat(k, G, axis=1), np.repeat(v, G, axis=1)
    np.testing.assert_allclose(o, _sdpa(q, kr, vr, mask, 1 / math.sqrt(D)), rtol=1e-12, atol=1e-12)


def test_identical_keys_give_mean_of_visible_values():
    """All scores equal -> uniform weights over the C + depth(i) + 1 visible slots."""
    T, C, D = 15, 5, 4
    g = np.random.default_rng(5)
    q = g.standard_normal((T, 1, D))
    k = np.tile(g.standard_normal((1, 1, D)), (C + T, 1, 1))
    v = g.standard_normal((C + T, 1, D))
    parents = syn.binary_tree(T)
    o = oracle.tree_attention(q, k, v, parents, C)
    for i in range(T):
        anc, a = [], i
        while True:
            anc.append(a)
            if a == 0:
                break
            a = (a - 1) // 2
        rows = list(range(C)) + [C + a for a in anc]
        np.testing.assert_allclose(o[i, 0], v[rows, 0].mean(axis=0), rtol=1e-12, atol=1e-12)


def test_relabelling_permutes_outputs():
    """Another topological order of the same tree permutes the outputs accordingly."""
    cfg = syn.shrink(syn.CONFIGS["llama2-7b-layer"], hq=2, hkv=2, d=16, ctx=(13, 13), vocab=50)
    w = syn.Workload(cfg, 3)
    par = w.trees[0]
    T = len(par)
    C = int(w.ctx_lens[0])
    g = np.random.default_rng(0)
    q, k, v = _rand_qkv(9, T, C, 2, 2, 16)
    o = oracle.tree_attention(q, k, v, par, C)
    # DFS preorder (children in reverse) is another topological order
    kids = oracle.children_sets(par)
    order, stack = [], [0]
    while stack:
        n = stack.pop()
        order.append(n)
        stack.extend(kids[n])
    new_of = {old: new for new, old in enumerate(order)}
    par2 = [-1 if par[old] < 0 else new_of[int(par[old])] for old in order]
    q2 = q[order]
    k2 = np.concatenate([k[:C], k[C + np.array(order)]])
    v2 = np.concatenate([v[:C], v[C + np.array(order)]])
    o2 = oracle.tree_attention(q2, k2, v2, par2, C)
    np.testing.assert_allclose(o2, o[order], rtol=1e-12, atol=1e-12)
    del g


# ----------------------------------------------------------------------------- top-k

def test_topk_worked_example():
    g = _load("topk_worked.json")
    row = np.array(g["row"])
    for c in g["cases"]:
        idx, val = oracle.topk(row, c["k"])
        assert idx.tolist() == c["idx"]
        assert val.tolist() == c["val"]


def test_topk_matches_lexsort_with_ties():
    g = np.random.default_rng(17)
    for trial in range(40):
        V = int(g.integers(1, 3000))
        row = np.round(g.standard_normal(V) * 3, 1)        # many exact ties
        row[g.integers(0, V, size=min(V, 5))] = 0.0
        row[g.integers(0, V, size=min(V, 5))] = -0.0
        k = int(g.integers(1, min(V, 16) + 1))
        order = np.lexsort((np.arange(V), -row))[:k]       # primary -value, secondary index
        idx, val = oracle.topk(row, k)
        assert idx.tolist() == order.tolist()
        assert np.array_equal(val, row[order])


def test_topk_brute_force_rank():
    """rank(j) = #{i : x_i > x_j or (x_i == x_j and i < j)}; top-k = ranks 0..k-1 in rank order."""
    g = np.random.default_rng(23)
    for _ in range(30):
        V = int(g.integers(1, 60))
        row = g.integers(-3, 4, size=V).astype(float)
        k = int(g.integers(1, V + 1))
        rank = [sum(1 for i in range(V) if row[i] > row[j] or (row[i] == row[j] and i < j)) for j in range(V)]
        expect = sorted(range(V), key=lambda j: rank[j])[:k]
        assert oracle.topk(row, k)[0].tolist() == expect


def test_topk_bf16_rows_widen_exactly():
    bits = syn.bf16_bits(np.random.default_rng(2).standard_normal((3, 500)).astype(np.float32))
    x = syn.widen(bits, "bf16")
    idx, val = oracle.topk_rows(x, 4)
    for r in range(3):
        order = np.lexsort((np.arange(500), -x[r]))[:4]
        assert idx[r].tolist() == order.tolist()


# ---------------------------------------------------------------------------- verify

def test_verify_worked_examples():
    for c in _load("verify_worked.json")["cases"]:
        I = oracle.eligible_edges(c["parents"], c["tokens"], c["target"])
        assert sorted(map(list, I)) == c["eligible_edges"]
        path, n, bonus = oracle.verify_greedy(c["parents"], c["tokens"], c["target"])
        assert path == c["path"] and n == c["accept_len"] and bonus == c["bonus"]


def _brute_force(parents, tokens, target):
    """Enumerate every root path (one per end node); keep eligible ones; longest, then lex-min."""
    best = None
    for end in range(len(parents)):
        path = [end]
        while parents[path[-1]] >= 0:
            path.append(parents[path[-1]])
        path.reverse()
        if all(tokens[c] == target[p] for p, c in zip(path, path[1:])):
            if best is None or len(path) > len(best) or (len(path) == len(best) and path < best):
                best = path
    return best, len(best), target[best[-1]]


def _recursive_trees(n):
    for tail in itertools.product(*[range(i) for i in range(1, n)]):
        yield [-1, *tail]


@pytest.mark.parametrize("n", [1, 2, 3, 4, 5, 6])
def test_verify_brute_force_exhaustive(n):
    for parents in _recursive_trees(n):
        for toks in itertools.product((0, 1), repeat=n - 1):
            tokens = [0, *toks]
            for target in itertools.product((0, 1), repeat=n):
                assert oracle.verify_greedy(parents, tokens, target) == _brute_force(parents, tokens, list(target))


def test_verify_brute_force_seven_nodes_exhaustive():
    """Every root path of every one of the 720 recursive trees with 7 nodes, under every
    binary token / target assignment (2^6 x 2^7 per tree, 5.9 million oracle calls): the
    brute force is vectorised over the assignments, and the trees are spread over worker
    processes started with spawn."""
    import multiprocessing as mp

    import _verify_brute_force as bf

    trees = list(bf.recursive_trees(7))
    assert len(trees) == 720
    workers = max(1, min(8, os.cpu_count() or 1))
    chunks = [trees[i::workers] for i in range(workers)]
    with mp.get_context("spawn").Pool(workers) as pool:
        counts = pool.map(bf.check_trees, chunks)
    assert sum(counts) == 720 * 2 ** 6 * 2 ** 7


def test_verify_brute_force_helper_catches_a_planted_mistake():
    """The vectorised brute force above is itself exercised against the plain one of this
    file on 6-node trees, and it rejects an oracle that prefers the largest sequence."""
    import _verify_brute_force as bf

    for parents in list(bf.recursive_trees(6))[::7]:
        tokens, target, best, lengths, paths = bf.brute_force_all_assignments(parents)
        for a in range(0, len(tokens), 97):
            want = _brute_force(parents, tokens[a].tolist(), target[a].tolist())
            assert (paths[int(best[a])], int(lengths[a]), int(target[a, int(best[a])])) == want
    parents = [-1, 0, 0]
    tokens, target, best, lengths, paths = bf.brute_force_all_assignments(parents)
    a = [i for i in range(len(tokens)) if tokens[i].tolist() == [0, 1, 1] and target[i, 0] == 1][0]
    assert paths[int(best[a])] == [0, 1]               # both children eligible: the smaller wins


@pytest.mark.parametrize("name", syn.CONFIG_ORDER)
def test_verify_invariants_on_workloads(name):
    cfg = syn.CONFIGS[name]
    if cfg.vocab > 40000:
        cfg = syn.shrink(cfg, vocab=4000)
    w = syn.Workload(cfg, 1)
    logits = syn.widen(w.logits, cfg.dtype)
    idx, _ = oracle.topk_rows(logits, 1)
    for b in range(cfg.batch):
        sl = w.nodes_of(b)
        par, tok, tgt = w.trees[b], w.tokens[sl], idx[sl, 0]
        path, n, bonus = oracle.verify_greedy(par, tok, tgt)
        d = oracle.depths(par)
        assert 1 <= n <= d.max() + 1                       # accepted edges <= tree depth
        assert path[0] == 0
        for p, c in zip(path, path[1:]):
            assert par[c] == p and tok[c] == tgt[p]        # a root path of eligible edges
        assert not any(tok[c] == tgt[path[-1]] for c in oracle.children_sets(par)[path[-1]])
        assert bonus == tgt[path[-1]]


# --------------------------------------------------------------------------- compact

def test_compact_worked_example():
    g = _load("compact_worked.json")
    slots = np.array(g["slots_before"])[:, None]
    new, new_ctx = oracle.kv_compact(slots, g["path"], g["ctx_len"])
    assert new_ctx == g["new_ctx"]
    assert new[:new_ctx, 0].tolist() == g["slots_after_prefix"]


def test_compact_matches_gather_and_keeps_prefix():
    g = np.random.default_rng(4)
    for _ in range(50):
        C, T = int(g.integers(0, 20)), int(g.integers(1, 30))
        parents = [-1] + [int(g.integers(0, i)) for i in range(1, T)]
        # a random root path
        end = int(g.integers(0, T))
        path = [end]
        while parents[path[-1]] >= 0:
            path.append(parents[path[-1]])
        path.reverse()
        cache = g.standard_normal((C + T + 3, 2, 4))
        new, nc = oracle.kv_compact(cache, path, C)
        assert nc == C + len(path)
        assert np.array_equal(new[:C], cache[:C])
        assert np.array_equal(new[C:nc], cache[C + np.array(path)])


# --------------------------------------------------------------------------- sampling verification

def _chi2_pvalue(counts, probs):
    """p-value of Pearson's chi-square statistic (library routine)."""
    stats = pytest.importorskip("scipy.stats")
    n = counts.sum()
    keep = probs > 0
    assert counts[~keep].sum() == 0            # a token of probability 0 is never emitted
    return stats.chisquare(counts[keep], n * probs[keep] / probs[keep].sum()).pvalue


def _emitted_first_token(parents, tokens, logits, u_acc, u_bon):
    path, alen, bonus, _ = oracle.verify_sampling(parents, tokens, logits, 1.0, u_acc, u_bon)
    return int(tokens[path[1]]) if alen > 1 else bonus


def test_sampling_worked_examples():
    """Hand-derived steps of Alg. 2 (tests/golden/sampling_worked.json): a rejection
    followed by renormalisation and an acceptance, a repeated candidate, and a full
    rejection with the bonus from the residual."""
    for c in _load("sampling_worked.json")["cases"]:
        logits = np.log(np.array(c["probs"], np.float64))
        path, n, bonus, margin = oracle.verify_sampling(c["parents"], np.array(c["tokens"]), logits, 1.0,
                                                       c["u_accept"], c["u_bonus"])
        assert (path, n, bonus) == (c["path"], c["accept_len"], c["bonus"]), c["why"]
        assert margin > 1e-3   # every decision is far from its threshold


def test_sampling_star_tree_emits_P():
    """App. E: trying the candidates in order with renormalisation after each rejection,
    and falling back to the residual, emits token i with probability exactly P_i.  The
    candidate tokens include a repeat (its second copy has probability 0 once the first is
    rejected)."""
    g = np.random.default_rng(11)
    V = 6
    row = g.normal(0.0, 1.0, V)
    P = oracle.softmax_row(row)
    parents = [-1, 0, 0, 0, 0]
    tokens = np.array([0, 2, 0, 2, 5])
    logits = np.tile(row, (5, 1))
    trials = 40000
    counts = np.zeros(V, np.int64)
    for _ in range(trials):
        u = g.random(5)
        counts[_emitted_first_token(parents, tokens, logits, u, g.random())] += 1
    assert _chi2_pvalue(counts, P) > 1e-4
    # and the acceptance of the first candidate is exactly P[token] (base case of App. E)
    g2 = np.random.default_rng(12)
    acc1 = sum(oracle.verify_sampling(parents, tokens, logits, 1.0, g2.random(5), 0.5)[0][1:2] == [1]
               for _ in range(20000))
    assert abs(acc1 / 20000 - P[2]) < 4 * math.sqrt(P[2] * (1 - P[2]) / 20000)


def test_sampling_leaf_root_bonus_is_P_and_temperature():
    g = np.random.default_rng(13)
    V = 5
    row = g.normal(0.0, 2.0, V)
    for temp in (1.0, 0.5):
        P = np.exp(row / temp - (row / temp).max())
        P /= P.sum()
        assert np.allclose(oracle.softmax_row(row, temp), P)
        counts = np.zeros(V, np.int64)
        for _ in range(30000):
            counts[oracle.verify_sampling([-1], [3], row[None, :], temp, [0.0], g.random())[2]] += 1
        assert _chi2_pvalue(counts, P) > 1e-4


def test_sampling_one_hot_reduces_to_greedy():
    """With all of P_v on argmax_v (a logit margin of 1e4) sampling accepts exactly the
    children whose token is the parent's argmax, so it walks the greedy path (siblings
    carry distinct tokens, as the workload generator guarantees)."""
    g = np.random.default_rng(14)
    V = 12
    for _ in range(200):
        T = int(g.integers(1, 40))
        parents = [-1] + [int(g.integers(0, i)) for i in range(1, T)]
        arg = g.integers(0, V, size=T)
        logits = g.normal(0.0, 1.0, (T, V))
        logits[np.arange(T), arg] += 1e4
        tokens = np.zeros(T, np.int64)
        for p, kids in enumerate(oracle.children_sets(parents)):
            perm = g.permutation(V)
            for j, c in enumerate(kids):   # distinct tokens among siblings, argmax[p] with probability 0.6
                tokens[c] = arg[p] if (j == 0 and g.random() < 0.6) else perm[(j + 1) % V]
        sig = oracle.children_sets(parents)
        for p, kids in enumerate(sig):     # keep siblings distinct after the substitution
            seen = set()
            for c in kids:
                while int(tokens[c]) in seen:
                    tokens[c] = (tokens[c] + 1) % V
                seen.add(int(tokens[c]))
        path, alen, bonus, _ = oracle.verify_sampling(parents, tokens, logits, 1.0, g.random(T), g.random())
        gpath, galen, gbonus = oracle.verify_greedy(parents, tokens, arg)
        assert (path, alen, bonus) == (gpath, galen, gbonus)


def test_sampling_invariants_on_random_trees():
    """Every accepted edge had positive probability, the bonus is not a token rejected at
    the last node and has positive probability, and the path fits in the tree."""
    g = np.random.default_rng(15)
    V = 20
    for _ in range(300):
        T = int(g.integers(1, 50))
        parents = [-1] + [int(g.integers(0, i)) for i in range(1, T)]
        logits = g.normal(0.0, 3.0, (T, V))
        tokens = g.integers(0, 4, size=T)            # few distinct tokens: repeats among siblings
        path, alen, bonus, margin = oracle.verify_sampling(parents, tokens, logits, 0.8, g.random(T), g.random())
        assert alen == len(path) and path[0] == 0 and alen - 1 <= int(oracle.depths(parents).max())
        for a, b in zip(path, path[1:]):
            assert parents[b] == a and oracle.softmax_row(logits[a], 0.8)[tokens[b]] > 0
        last = path[-1]
        rejected = {int(tokens[c]) for c in oracle.children_sets(parents)[last]}
        assert bonus not in rejected or len(rejected) == V
        assert oracle.softmax_row(logits[last], 0.8)[bonus] > 0 and margin >= 0


# ---------------------------------------------------------------------------
# Draft tree update (Sec. 3.1 Progressive Expansion, Width Control, Stepping
# Mechanism; Alg. 1 step 3)
# ---------------------------------------------------------------------------

def test_draft_update_worked_examples():
    for case in _load("draft_update_worked.json")["cases"]:
        got = oracle.draft_tree_update(case["parents"], case["tokens"], case["drafts"], case["expand"],
                                       case["width"], case["max_depth"], case["capacity"])
        for name, arr in zip(("new_parents", "new_tokens", "new_depths", "old_to_new"), got):
            assert arr.tolist() == case[name], (case["why"], name)


class _TrieNode:
    """A draft-forest node as a token-keyed trie entry with a creation stamp."""

    def __init__(self, token, stamp, origin):
        self.token, self.stamp, self.origin, self.kids = token, stamp, origin, []


def _trie_update(parents, tokens, drafts, expand, width, max_depth, capacity):
    """The same step written over nested trie objects instead of index arrays:
    expansion walks the original nodes by stamp, a child is found by token, a stepped
    subtree is re-rooted at kids[0] (its earliest stamp), and the survivors are
    flattened by stamp."""
    nodes = [_TrieNode(int(t), i, i) for i, t in enumerate(tokens)]
    roots = []
    for i, p in enumerate(parents):
        (roots if p == -1 else nodes[p].kids).append(nodes[i])
    count = len(nodes)
    for v in list(nodes):
        for d in drafts[v.origin][:expand]:
            if any(c.token == int(d) for c in v.kids) or len(v.kids) >= width or count >= capacity:
                continue
            v.kids.append(_TrieNode(int(d), count, -1))
            count += 1

    def height(n):
        return 1 + max((height(c) for c in n.kids), default=0)

    roots = [r.kids[0] if height(r) > max_depth else r for r in roots]
    out = []                                        # (stamp, node, parent node or None)

    def collect(n, parent):
        out.append((n.stamp, n, parent))
        for c in n.kids:
            collect(c, n)

    for r in roots:
        collect(r, None)
    out.sort(key=lambda e: e[0])
    index = {id(n): k for k, (_, n, _) in enumerate(out)}
    new_par = [-1 if par is None else index[id(par)] for _, _, par in out]
    new_tok = [n.token for _, n, _ in out]
    new_dep = []
    for k, p in enumerate(new_par):
        new_dep.append(1 if p == -1 else new_dep[p] + 1)
    old_to_new = [-1] * len(parents)
    for k, (_, n, _) in enumerate(out):
        if n.origin >= 0:
            old_to_new[n.origin] = k
    return new_par, new_tok, new_dep, old_to_new


def _random_forest(g, T, n_tokens):
    parents = []
    for i in range(T):
        parents.append(-1 if (i == 0 or g.random() < 0.15) else int(g.integers(0, i)))
    tokens = []
    kids_tokens = {}
    for i, p in enumerate(parents):      # siblings carry distinct tokens, as in a trie
        used = kids_tokens.setdefault(p, set()) if p >= 0 else set()
        t = int(g.integers(0, n_tokens))
        while t in used and len(used) < n_tokens:
            t = (t + 1) % n_tokens
        if t in used:                    # every token taken: a fresh one past the range
            t = n_tokens + len(used)
        used.add(t)
        tokens.append(t)
    return parents, tokens


def test_draft_update_matches_trie_formulation():
    g = np.random.default_rng(21)
    for _ in range(600):
        T = int(g.integers(1, 30))
        parents, tokens = _random_forest(g, T, 12)
        expand = int(g.integers(0, 4))
        drafts = g.integers(0, 12, size=(T, 4))
        width = int(g.integers(0, 5))
        max_depth = int(g.integers(1, 8))
        capacity = T + int(g.integers(0, 3 * T + 2))
        got = oracle.draft_tree_update(parents, tokens, drafts, expand, width, max_depth, capacity)
        want = _trie_update(parents, tokens, drafts, expand, width, max_depth, capacity)
        for a, b in zip(got, want):
            assert a.tolist() == list(b)


def test_draft_update_invariants():
    """The result is a forest in creation order; no subtree is deeper than d_max when the
    input was within it; width and sibling-token distinctness are preserved; every kept
    node's root-to-node token path is its old path, less the stepped seed's token."""
    g = np.random.default_rng(22)
    for _ in range(400):
        T = int(g.integers(1, 40))
        parents, tokens = _random_forest(g, T, 30)
        dep = []
        for p in parents:
            dep.append(1 if p == -1 else dep[p] + 1)
        max_depth = max(dep) + int(g.integers(0, 2))
        width = 8
        drafts = g.integers(0, 30, size=(T, 3))
        new_par, new_tok, new_dep, o2n = oracle.draft_tree_update(parents, tokens, drafts, 2, width, max_depth, 128)
        oracle.check_forest(new_par)
        assert int(new_dep.max()) <= max_depth
        for v in range(len(new_par)):
            kids = [i for i in range(len(new_par)) if new_par[i] == v]
            assert len(kids) <= width
            assert len({int(new_tok[i]) for i in kids}) == len(kids)

        def path(par, tok, i):
            out = []
            while i != -1:
                out.append(int(tok[i]))
                i = par[i]
            return out[::-1]

        for j, k in enumerate(o2n):
            if k < 0:
                continue
            old, new = path(parents, tokens, j), path(list(new_par), new_tok, int(k))
            assert old == new or old[1:] == new


def test_draft_update_identity_and_sliding_window():
    """With nothing to add and no depth limit the step is the identity; on a chain fed
    the next token of a sequence every step, the stepping mechanism keeps exactly the
    last d_max tokens (a sliding window, Sec. 3.1 and Fig. 3)."""
    g = np.random.default_rng(23)
    parents, tokens = _random_forest(g, 25, 9)
    got = oracle.draft_tree_update(parents, tokens, np.zeros((25, 1), np.int64), 0, 4, 99, 64)
    assert got[0].tolist() == parents and got[1].tolist() == tokens and got[3].tolist() == list(range(25))
    seq = list(g.integers(0, 1000, size=40))
    d_max = 6
    par, tok = [-1], [int(seq[0])]
    for step in range(1, 40):
        drafts = [[tok[i + 1]] if i + 1 < len(tok) else [int(seq[step])] for i in range(len(tok))]
        par, tok, dep, _ = oracle.draft_tree_update(par, tok, drafts, 1, 1, d_max, 64)
        par, tok = par.tolist(), tok.tolist()
        assert tok == [int(x) for x in seq[max(0, step + 1 - d_max):step + 1]]
        assert par == [-1] + list(range(len(tok) - 1)) and dep.tolist() == list(range(1, len(tok) + 1))


# ---------------------------------------------------------------------------
# Candidate pool (Sec. 3.1 "Draft Extraction via Merging"; Sec. 3.2; Alg. 1 steps 1, 4)
# ---------------------------------------------------------------------------

def test_pool_worked_example():
    gold = _load("candidate_pool_worked.json")
    pool = oracle.CandidatePool()
    for step in gold["steps"]:
        pool.merge_forest(step["parents"], step["tokens"])
        assert pool.size() == step["pool_size"], step["why"]
        for r in step["retrieve"]:
            par, tok = pool.retrieve(r["root"], r["width"], r["max_depth"], r["max_nodes"])
            assert par.tolist() == r["parents"] and tok.tolist() == r["tokens"], (step["why"], r)


def _path_set_pool(forests):
    """The pool as a set of token paths with first-insertion keys: every (v, u) pair with u
    in v's subtree inserts the path token(v) .. token(u); a path first inserted at step s by
    the pair (v, u) gets the key (s, v, u)."""
    first = {}
    for s, (parents, tokens) in enumerate(forests):
        for u in range(len(parents)):
            chain = []
            a = u
            while a != -1:
                chain.append(a)
                a = parents[a]
            chain.reverse()                    # seed .. u
            for k, v in enumerate(chain):
                path = tuple(int(tokens[x]) for x in chain[k:])
                first[path] = min(first.get(path, (s, v, u)), (s, v, u))
    return first


def _path_set_retrieve(first, root, width, max_depth, max_nodes):
    """Breadth-first over the path set: the children of a path are its one-token
    extensions, the `width` smallest first-insertion keys first."""
    if (root,) not in first:
        return [-1], [root]
    ext_of = {}
    for path, key in first.items():
        if len(path) > 1:
            ext_of.setdefault(path[:-1], []).append((key, path))
    parents, tokens, paths = [-1], [root], [(root,)]
    frontier, depth = [0], 1
    while frontier and depth < max_depth and len(tokens) < max_nodes:
        nxt = []
        for idx in frontier:
            p = paths[idx]
            ext = sorted(ext_of.get(p, []))
            for _, path in ext[:width]:
                if len(tokens) >= max_nodes:
                    break
                parents.append(idx)
                tokens.append(path[-1])
                paths.append(path)
                nxt.append(len(tokens) - 1)
        frontier, depth = nxt, depth + 1
    return parents, tokens


def test_pool_matches_path_set_formulation():
    g = np.random.default_rng(31)
    for _ in range(40):
        pool = oracle.CandidatePool()
        forests = []
        for step in range(int(g.integers(1, 6))):
            parents, tokens = _random_forest(g, int(g.integers(1, 25)), 6)
            pool.merge_forest(parents, tokens)
            forests.append((parents, tokens))
            first = _path_set_pool(forests)
            assert pool.size() == len(first)
            for root in range(7):
                width, max_depth, max_nodes = int(g.integers(1, 5)), int(g.integers(1, 7)), int(g.integers(1, 40))
                par, tok = pool.retrieve(root, width, max_depth, max_nodes)
                want = _path_set_retrieve(first, root, width, max_depth, max_nodes)
                assert (par.tolist(), tok.tolist()) == want


def test_pool_idempotent_and_chain():
    """Merging the same forest again adds nothing; a chain t1..tn gives every ti an entry
    holding the rest of the chain."""
    g = np.random.default_rng(32)
    parents, tokens = _random_forest(g, 30, 8)
    pool = oracle.CandidatePool()
    pool.merge_forest(parents, tokens)
    size = pool.size()
    before = [pool.retrieve(r, 3, 5, 50) for r in range(8)]
    pool.merge_forest(parents, tokens)
    assert pool.size() == size
    for r in range(8):
        a, b = before[r], pool.retrieve(r, 3, 5, 50)
        assert a[0].tolist() == b[0].tolist() and a[1].tolist() == b[1].tolist()
    seq = [int(x) for x in g.permutation(100)[:12]]
    chain = oracle.CandidatePool()
    chain.merge_forest([-1] + list(range(11)), seq)
    for i, t in enumerate(seq):
        par, tok = chain.retrieve(t, 4, 99, 99)
        assert tok.tolist() == seq[i:] and par.tolist() == [-1] + list(range(len(seq) - i - 1))


# ---------------------------------------------------------------------------
# Tree positions and the rotary encoding (Sec. 3.1 "Tree Construction")
# ---------------------------------------------------------------------------

def test_tree_positions_closed_forms():
    """A chain sits at C .. C + T - 1 (ordinary causal positions), a star's leaves all at
    C + 1, and a node's position is its parent's plus one."""
    assert oracle.tree_positions([-1, 0, 1, 2, 3], 100).tolist() == [100, 101, 102, 103, 104]
    assert oracle.tree_positions([-1, 0, 0, 0], 7).tolist() == [7, 8, 8, 8]
    g = np.random.default_rng(41)
    parents = [-1] + [int(g.integers(0, i)) for i in range(1, 60)]
    pos = oracle.tree_positions(parents, 33)
    assert pos[0] == 33 and all(pos[i] == pos[parents[i]] + 1 for i in range(1, 60))


def test_rope_defining_properties():
    """RoFormer's rotation: position 0 is the identity, norms are kept, rotations compose
    (rope(rope(x, a), b) = rope(x, a + b)), and q.k after encoding depends only on the
    offset between the two positions."""
    g = np.random.default_rng(42)
    x = g.normal(size=(5, 3, 64))
    y = g.normal(size=(5, 3, 64))
    base = 10000.0
    assert np.allclose(oracle.rope(x, np.zeros(5), base), x)
    p = g.integers(0, 5000, size=5)
    r = oracle.rope(x, p, base)
    assert np.allclose(np.linalg.norm(r, axis=-1), np.linalg.norm(x, axis=-1))
    q = g.integers(0, 5000, size=5)
    assert np.allclose(oracle.rope(r, q, base), oracle.rope(x, p + q, base))
    shift = 1234
    d1 = np.sum(oracle.rope(x, p, base) * oracle.rope(y, q, base), axis=-1)
    d2 = np.sum(oracle.rope(x, p + shift, base) * oracle.rope(y, q + shift, base), axis=-1)
    assert np.allclose(d1, d2)
    # the lowest pair turns by exactly the position (angle pos * base^0) and the rest slower
    e = np.zeros((1, 1, 64))
    e[0, 0, 0] = 1.0
    out = oracle.rope(e, [3], base)[0, 0]
    assert np.isclose(out[0], np.cos(3.0)) and np.isclose(out[32], np.sin(3.0))
    # pair 5 of 32 turns by 3 * 10000^(-10/64) = 3 * 10^-0.625 = 0.71141211 rad
    e = np.zeros((1, 1, 64))
    e[0, 0, 5] = 1.0
    out = oracle.rope(e, [3], base)[0, 0]
    assert np.isclose(out[5], 0.7574406580936761) and np.isclose(out[37], 0.652904012444876)
    assert np.count_nonzero(np.abs(out) > 1e-12) == 2


# ---------------------------------------------------------------------------
# LM head with top-k
# ---------------------------------------------------------------------------

def test_lm_head_worked_example_and_brute_force():
    """A 2-node, 5-token example worked by hand, and random cases against a brute-force
    dot product per (node, token) with a sort by (-value, index)."""
    h = [[1.0, 2.0], [0.5, -1.0]]
    w = [[1, 0], [0, 1], [1, 1], [-1, 0], [2, -1]]
    # node 0: logits 1, 2, 3, -1, 0 -> top-2 tokens 2, 1; node 1: 0.5, -1, -0.5, -0.5, 2 -> 4, 0
    idx, val = oracle.lm_head_topk(h, w, 2)
    assert idx.tolist() == [[2, 1], [4, 0]] and val.tolist() == [[3.0, 2.0], [2.0, 0.5]]
    idx, _ = oracle.lm_head_topk([[0.0, 1.0]], [[1, 2], [3, 2], [5, 2]], 3)   # a three-way tie
    assert idx.tolist() == [[0, 1, 2]]
    g = np.random.default_rng(51)
    for _ in range(20):
        N, d, V = int(g.integers(1, 6)), int(g.integers(1, 9)), int(g.integers(1, 40))
        k = min(V, int(g.integers(1, 6)))
        hh = g.integers(-3, 4, size=(N, d)).astype(float)
        ww = g.integers(-3, 4, size=(V, d)).astype(float)   # small integers: many exact ties
        idx, val = oracle.lm_head_topk(hh, ww, k)
        for n in range(N):
            logits = [sum(hh[n, j] * ww[t, j] for j in range(d)) for t in range(V)]
            order = sorted(range(V), key=lambda t: (-logits[t], t))[:k]
            assert idx[n].tolist() == order and val[n].tolist() == [logits[t] for t in order]
