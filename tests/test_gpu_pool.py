"""Candidate pool on the GPU against the oracle (Sec. 3.1 "Draft Extraction via Merging";
Sec. 3.2; Alg. 1 steps 1 and 4).  Integer work: node counts and every retrieved tree must
be bit-exact."""
import numpy as np
import pytest
import torch

import oracle
from paper_2607_10661_gb300 import ptd

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    import __graft_entry__

    __graft_entry__.build()


def _forest(g, T, n_tokens, seed_p=0.15):
    parents, tokens, kid_tokens = [], [], {}
    for i in range(T):
        p = -1 if (i == 0 or g.random() < seed_p) else int(g.integers(0, i))
        used = kid_tokens.setdefault(p, set()) if p >= 0 else set()
        t = int(g.integers(0, n_tokens))
        while t in used and len(used) < n_tokens:
            t = (t + 1) % n_tokens
        if t in used:
            t = n_tokens + len(used)
        used.add(t)
        parents.append(p)
        tokens.append(t)
    return parents, tokens


def _dev(x):
    return torch.tensor(x, dtype=torch.int32, device="cuda")


class _Outs:
    def __init__(self, n=128):
        self.count = torch.zeros(1, dtype=torch.int32, device="cuda")
        self.parents = torch.empty(n, dtype=torch.int32, device="cuda")
        self.tokens = torch.empty(n, dtype=torch.int32, device="cuda")


def _retrieve(pool, root, width, max_depth, max_nodes, o):
    assert pool.retrieve(_dev([root]), width, max_depth, max_nodes, o.count, o.parents, o.tokens) == 1
    n = int(o.count.item())
    par, tok = o.parents.cpu().numpy(), o.tokens.cpu().numpy()
    assert (par[n:max_nodes] == -1).all() and (tok[n:max_nodes] == -1).all()
    return par[:n].tolist(), tok[:n].tolist()


@pytest.mark.parametrize("capacity,n_tokens", [(1 << 16, 6), (1 << 10, 40), (1 << 20, 500)])
def test_merge_and_retrieve_match_oracle(capacity, n_tokens):
    """Random forests merged step after step (small capacities exercise long probe runs),
    every entry retrieved with random budgets after every step."""
    g = np.random.default_rng(capacity)
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    o = _Outs()
    for trial in range(4):
        pool, ref = ptd.CandidatePool(capacity), oracle.CandidatePool()
        for step in range(8):
            parents, tokens = _forest(g, int(g.integers(1, 129 if capacity >= 1 << 16 else 33)), n_tokens)
            pairs = 0
            for u in range(len(parents)):      # pairs (v, u): the merge's bound on new nodes
                a = u
                while a != -1:
                    pairs += 1
                    a = parents[a]
            if pool.size() + pairs > capacity // 2:
                break
            ref.merge_forest(parents, tokens)
            assert pool.merge(step, _dev([len(parents)]), _dev(parents), _dev(tokens), status) == 1
            assert pool.size() == ref.size()
            roots = sorted(set(tokens))[:12] + [n_tokens + 1000]
            for root in roots:
                width, max_depth, max_nodes = int(g.integers(1, 9)), int(g.integers(1, 9)), int(g.integers(1, 129))
                par, tok = ref.retrieve(root, width, max_depth, max_nodes)
                assert _retrieve(pool, root, width, max_depth, max_nodes, o) == (par.tolist(), tok.tolist())
    assert int(status.item()) == 0


def test_chain_and_idempotent_merge():
    g = np.random.default_rng(5)
    seq = [int(x) for x in g.permutation(1000)[:40]]
    pool = ptd.CandidatePool(1 << 12)
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    parents = [-1] + list(range(39))
    pool.merge(0, _dev([40]), _dev(parents), _dev(seq), status)
    n = pool.size()
    assert n == 40 * 41 // 2
    pool.merge(1, _dev([40]), _dev(parents), _dev(seq), status)
    assert pool.size() == n and int(status.item()) == 0
    o = _Outs()
    for i in (0, 7, 39):
        par, tok = _retrieve(pool, seq[i], 8, 99, 128, o)
        assert tok == seq[i:] and par == [-1] + list(range(39 - i))


def test_pool_full_and_invalid_forest_leave_the_pool_unchanged():
    g = np.random.default_rng(6)
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    pool = ptd.CandidatePool(64)
    parents, tokens = _forest(g, 30, 10)
    pool.merge(0, _dev([30]), _dev(parents), _dev(tokens), status, max_load=20)   # 30+ pairs > 20
    assert int(status.item()) == ptd.POOL_FULL and pool.size() == 0
    status.zero_()
    bad = list(parents)
    bad[4] = 17
    pool.merge(1, _dev([30]), _dev(bad), _dev(tokens), status)
    assert int(status.item()) == ptd.INVALID_TREE and pool.size() == 0
    o = _Outs()
    assert _retrieve(pool, tokens[0], 4, 6, 16, o) == ([-1], [tokens[0]])


def test_device_loop_update_merge_retrieve():
    """Ten steps on the device: the draft forest grows and steps (ptd_draft_tree_update),
    its subtrees join the pool, and the candidate tree of the forest's first seed token is
    retrieved, against the oracle doing the same on the host."""
    g = np.random.default_rng(7)
    cap_f, V = 96, 30
    parents, tokens = _forest(g, 12, V)
    cnt = _dev([len(parents)])
    par = torch.full((1, cap_f), -1, dtype=torch.int32, device="cuda")
    tok = torch.full((1, cap_f), -1, dtype=torch.int32, device="cuda")
    par[0, :len(parents)] = _dev(parents)
    tok[0, :len(tokens)] = _dev(tokens)
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    pool, ref = ptd.CandidatePool(1 << 14), oracle.CandidatePool()
    o = _Outs()
    for step in range(10):
        dr = g.integers(0, V, size=(cap_f, 2))
        outs = [torch.empty_like(x) for x in (cnt, par, tok, par, par)]
        ptd.draft_tree_update(cnt, par, tok, torch.tensor(dr, dtype=torch.int32, device="cuda"), 1, 3, 5, cap_f,
                              *outs, status)
        p2, t2, _, _ = oracle.draft_tree_update(parents, tokens, dr[:max(1, len(parents))], 1, 3, 5, cap_f)
        parents, tokens = p2.tolist(), t2.tolist()
        cnt, par, tok = outs[0], outs[1], outs[2]
        pool.merge(step, cnt, par[0], tok[0], status)
        ref.merge_forest(parents, tokens)
        got = _retrieve(pool, tokens[0], 4, 6, 64, o)
        want = ref.retrieve(tokens[0], 4, 6, 64)
        assert got == (want[0].tolist(), want[1].tolist())
        assert pool.size() == ref.size()
    assert int(status.item()) == 0
