"""Exhaustive brute force of greedy verification on small trees (test helper, CPU only).

For one parent array, every assignment of binary draft tokens (the root's token fixed at
0) and binary greedy targets is enumerated at once with numpy: an edge (p, c) is eligible
when token[c] == target[p] (the set I of Sec. 3.2); every node ends exactly one root
path; among the paths whose edges are all eligible the longest wins, ties going to the
lexicographically smallest node sequence; the bonus token is the target of the path's last
node.  The oracle is then called on every assignment and must agree.

Kept in a module of its own (numpy and the oracle only) so that worker processes started
with `spawn` import it quickly.
"""
from __future__ import annotations

import itertools

import numpy as np

import oracle


def recursive_trees(n: int):
    """Every parent array of n nodes in topological order (parents[i] < i): (n-1)! of them."""
    for tail in itertools.product(*[range(i) for i in range(1, n)]):
        yield [-1, *tail]


def brute_force_all_assignments(parents):
    """(tokens [A, n], target [A, n], end node [A], path length [A]) over all
    A = 2^(n-1) * 2^n binary assignments, from the definition by enumeration."""
    n = len(parents)
    toks = np.array(list(itertools.product((0, 1), repeat=n - 1)), np.int64).reshape(-1, n - 1)
    tgts = np.array(list(itertools.product((0, 1), repeat=n)), np.int64)
    tokens = np.concatenate([np.zeros((len(toks), 1), np.int64), toks], axis=1)
    tokens = np.repeat(tokens, len(tgts), axis=0)
    target = np.tile(tgts, (len(toks), 1))
    elig = np.ones(tokens.shape, bool)
    for c in range(1, n):
        elig[:, c] = tokens[:, c] == target[:, parents[c]]
    paths = []
    for end in range(n):
        path = [end]
        while parents[path[-1]] >= 0:
            path.append(parents[path[-1]])
        paths.append(path[::-1])
    order = sorted(range(n), key=lambda e: (-len(paths[e]), paths[e]))
    best = np.full(len(tokens), -1, np.int64)
    for e in order:
        ok = np.all(elig[:, paths[e][1:]], axis=1) if len(paths[e]) > 1 else np.ones(len(tokens), bool)
        take = ok & (best < 0)
        best[take] = e
    lengths = np.array([len(paths[e]) for e in best], np.int64)
    return tokens, target, best, lengths, paths


def check_tree_exhaustively(parents) -> int:
    """Compare the oracle with the brute force on every assignment of one tree; returns the
    number of assignments checked, raises AssertionError on the first disagreement."""
    tokens, target, best, lengths, paths = brute_force_all_assignments(parents)
    for a in range(len(tokens)):
        got = oracle.verify_greedy(parents, tokens[a], target[a])
        e = int(best[a])
        want = (paths[e], int(lengths[a]), int(target[a, e]))
        assert got == want, (parents, tokens[a].tolist(), target[a].tolist(), got, want)
    return len(tokens)


def check_trees(tree_list) -> int:
    return sum(check_tree_exhaustively(p) for p in tree_list)
