"""The PTD decoding loop's bookkeeping on the GPU against the oracle, step after step
(Alg. 1 steps 1 and 3-6): retrieve the candidate tree of the current token from the pool,
verify the tree formed by it and the draft forest (top-k of the nodes' logits, greedy
verification), grow and step the draft forest by the top-k drafts, merge it into the pool,
continue from the bonus token.  Each side evolves its own state (the GPU from its kernels'
outputs, the oracle from its own); only the per-step logits are shared, and they are a
seeded function of the verification tree, so any divergence shows up as a mismatch."""
import numpy as np
import pytest
import torch

import oracle
from paper_2607_10661_gb300 import ptd

pytestmark = pytest.mark.gpu

V = 50                  # vocabulary
K = 4                   # top-k
WIDTH, DEPTH = 3, 4     # draft forest: width control and depth limit (Sec. 3.1)
CAP_F = 48              # draft forest capacity
C_W, C_D, C_N = 3, 4, 24   # candidate-tree retrieval budgets


@pytest.fixture(scope="module", autouse=True)
def _built():
    import __graft_entry__

    __graft_entry__.build()


def _compose(cand_par, cand_tok, f_par, f_tok):
    """Verification tree: the candidate tree (its node 0 is the current token), then the
    draft forest with its seeds hung under node 0.  Returns parents, tokens, offset of F."""
    off = len(cand_par)
    par = list(cand_par) + [0 if p == -1 else off + p for p in f_par]
    tok = list(cand_tok) + list(f_tok)
    return par, tok, off


def _logits(step, par, tok):
    """A seeded 'language model': node v's row peaks (+4) on (7 * token(v) + 3) mod V."""
    g = np.random.default_rng(1000 + step)
    x = g.normal(0.0, 1.0, (len(par), V)).astype(np.float32)
    for v, t in enumerate(tok):
        x[v, (7 * int(t) + 3) % V] += 4.0
    return x


def _dev(a):
    return torch.tensor(np.asarray(a), dtype=torch.int32, device="cuda")


def test_ptd_loop_matches_oracle():
    g = np.random.default_rng(5)
    seeds = [int(t) for t in g.choice(V, 5, replace=False)]
    x0 = int(g.integers(V))
    # ---- oracle state
    o_par, o_tok = [-1] * len(seeds), list(seeds)
    o_pool = oracle.CandidatePool()
    o_x = x0
    # ---- GPU state
    dev = "cuda"
    f_cnt = _dev([len(seeds)])
    f_par = torch.full((1, CAP_F), -1, dtype=torch.int32, device=dev)
    f_tok = torch.full((1, CAP_F), -1, dtype=torch.int32, device=dev)
    f_par[0, :len(seeds)] = _dev([-1] * len(seeds))
    f_tok[0, :len(seeds)] = _dev(seeds)
    pool = ptd.CandidatePool(1 << 14)
    x_dev = _dev([x0])
    status = torch.zeros(1, dtype=torch.int32, device=dev)
    rc = torch.zeros(1, dtype=torch.int32, device=dev)
    rp = torch.empty(C_N, dtype=torch.int32, device=dev)
    rt = torch.empty(C_N, dtype=torch.int32, device=dev)
    accepted_total = 0
    for step in range(12):
        # Alg. 1 step 1: candidate tree of the current token
        c_par, c_tok = o_pool.retrieve(o_x, C_W, C_D, C_N)
        pool.retrieve(x_dev, C_W, C_D, C_N, rc, rp, rt)
        n_c = int(rc.item())
        gc_par, gc_tok = rp[:n_c].cpu().tolist(), rt[:n_c].cpu().tolist()
        assert (gc_par, gc_tok) == (c_par.tolist(), c_tok.tolist()), step
        # the verification tree, each side from its own state
        n_f = int(f_cnt.item())
        gf_par, gf_tok = f_par[0, :n_f].cpu().tolist(), f_tok[0, :n_f].cpu().tolist()
        assert (gf_par, gf_tok) == (list(o_par), list(o_tok)), step
        par, tok, off = _compose(c_par.tolist(), c_tok.tolist(), o_par, o_tok)
        gpar, gtok, goff = _compose(gc_par, gc_tok, gf_par, gf_tok)
        lg = _logits(step, par, tok)
        # top-k (Sec. 3.1 drafts, Sec. 3.2 verification tokens) and greedy verification
        idx_ref, _ = oracle.topk_rows(lg, K)
        path, alen, bonus = oracle.verify_greedy(par, tok, idx_ref[:, 0])
        T = len(gpar)
        logits = torch.tensor(_logits(step, gpar, gtok), device=dev)
        idx = torch.empty((T, K), dtype=torch.int32, device=dev)
        val = torch.empty((T, K), dtype=torch.float32, device=dev)
        ptd.topk_draft(logits, K, idx, val)
        tree = ptd.Tree(_dev([0, T]), _dev(gpar), _dev([0]), T, 0)
        acc = torch.full((1, T), -1, dtype=torch.int32, device=dev)
        alen_d = torch.zeros(1, dtype=torch.int32, device=dev)
        bonus_d = torch.zeros(1, dtype=torch.int32, device=dev)
        ptd.verify_greedy(tree, _dev(gtok), idx, K, acc, alen_d, bonus_d, status)
        assert np.array_equal(idx.cpu().numpy(), idx_ref), step
        assert int(alen_d.item()) == alen and acc[0, :alen].cpu().tolist() == path and int(bonus_d.item()) == bonus
        accepted_total += alen
        # Alg. 1 step 3: the draft forest grows by its nodes' top-1 and is stepped
        drafts_ref = idx_ref[off:off + len(o_par)]
        o_par, o_tok, _, _ = oracle.draft_tree_update(o_par, o_tok, drafts_ref, 1, WIDTH, DEPTH, CAP_F)
        o_par, o_tok = o_par.tolist(), o_tok.tolist()
        drafts = torch.full((CAP_F, K), -1, dtype=torch.int32, device=dev)
        drafts[:n_f] = idx[goff:goff + n_f]
        outs = [torch.empty_like(f_cnt), torch.empty_like(f_par), torch.empty_like(f_tok), torch.empty_like(f_par),
                torch.empty_like(f_par)]
        ptd.draft_tree_update(f_cnt, f_par, f_tok, drafts, 1, WIDTH, DEPTH, CAP_F, *outs, status)
        f_cnt, f_par, f_tok = outs[0], outs[1], outs[2]
        # Alg. 1 step 4: every subtree of the new forest joins the pool
        o_pool.merge_forest(o_par, o_tok)
        pool.merge(step, f_cnt, f_par[0], f_tok[0], status)
        assert pool.size() == o_pool.size(), step
        # Alg. 1 step 6: the next current token is the bonus token
        o_x = bonus
        x_dev = bonus_d
    assert int(status.item()) == 0
    assert accepted_total > 12     # some steps accepted more than the root
