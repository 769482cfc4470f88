"""ptd_draft_tree_update on the GPU against the oracle (Sec. 3.1 Progressive Expansion,
Width Control, Stepping Mechanism; Alg. 1 step 3).  Integer work: every output must be
bit-exact, including the -1 fill past each forest's count."""
import numpy as np
import pytest
import torch

import oracle
from paper_2607_10661_gb300 import ptd
from paper_2607_10661_gb300 import synthetic as syn

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
        if t in used:                    # every token taken: a fresh one past the range
            t = n_tokens + len(used)
        used.add(t)
        parents.append(p)
        tokens.append(t)
    return parents, tokens


def _run(forests, drafts, expand, width, max_depth, capacity, stride=None, dstride=None):
    """forests: list of (parents, tokens); drafts: list of [T, >= expand] arrays."""
    B = len(forests)
    stride = stride or max(1, max(len(p) for p, _ in forests))
    dstride = dstride or max(1, expand)
    dev = "cuda"
    par = torch.full((B, stride), -7, dtype=torch.int32)
    tok = torch.full((B, stride), -7, dtype=torch.int32)
    dr = torch.full((B * stride, dstride), -5, dtype=torch.int32)
    cnt = torch.zeros(B, dtype=torch.int32)
    for b, (p, t) in enumerate(forests):
        cnt[b] = len(p)
        par[b, :len(p)] = torch.tensor(p, dtype=torch.int32)
        tok[b, :len(t)] = torch.tensor(t, dtype=torch.int32)
        d = np.asarray(drafts[b], np.int64)
        if len(p):
            dr[b * stride:b * stride + len(p), :d.shape[1]] = torch.tensor(d[:, :dstride], dtype=torch.int32)
    ins = [x.to(dev) for x in (cnt, par, tok, dr)]
    outs = dict(count=torch.full((B,), -9, dtype=torch.int32, device=dev),
                parents=torch.full((B, capacity), -9, dtype=torch.int32, device=dev),
                tokens=torch.full((B, capacity), -9, dtype=torch.int32, device=dev),
                depths=torch.full((B, capacity), -9, dtype=torch.int32, device=dev),
                o2n=torch.full((B, stride), -9, dtype=torch.int32, device=dev))
    status = torch.zeros(1, dtype=torch.int32, device=dev)
    n = ptd.draft_tree_update(ins[0], ins[1], ins[2], ins[3], expand, width, max_depth, capacity, outs["count"],
                              outs["parents"], outs["tokens"], outs["depths"], outs["o2n"], status)
    assert n == 1
    torch.cuda.synchronize()
    return {k: v.cpu().numpy() for k, v in outs.items()}, int(status.item()), stride


def _check(got, forests, drafts, expand, width, max_depth, capacity, stride):
    for b, (p, t) in enumerate(forests):
        want = oracle.draft_tree_update(p, t, np.asarray(drafts[b])[:, :expand] if len(p) else np.zeros((0, 1)),
                                        expand, width, max_depth, capacity)
        m = len(want[0])
        assert got["count"][b] == m, b
        for key, w in zip(("parents", "tokens", "depths"), want[:3]):
            assert got[key][b, :m].tolist() == w.tolist(), (b, key)
            assert (got[key][b, m:] == -1).all(), (b, key)
        assert got["o2n"][b, :len(p)].tolist() == want[3].tolist(), b
        assert (got["o2n"][b, len(p):stride] == -1).all(), b


@pytest.mark.parametrize("seed", [1, 2, 3])
def test_random_forests_match_oracle(seed):
    g = np.random.default_rng(seed)
    for _ in range(6):
        B = int(g.integers(1, 9))
        expand = int(g.integers(1, 5))
        width = int(g.integers(0, 6))
        max_depth = int(g.integers(1, 9))
        capacity = int(g.integers(40, 129))
        forests = [_forest(g, int(g.integers(0, 41)), 8) for _ in range(B)]
        drafts = [g.integers(0, 8, size=(max(1, len(p)), 6)) for p, _ in forests]
        got, status, stride = _run(forests, drafts, expand, width, max_depth, capacity)
        assert status == 0
        _check(got, forests, drafts, expand, width, max_depth, capacity, stride)


def test_step_tree_with_topk_drafts():
    """The Llama-3-8B-shaped step's 63-node tree (one seed) grown by the top-1 of its own
    logits' top-k, width 4, depth 6 (the paper's best setting, Fig. 6)."""
    w = syn.Workload(syn.shrink(syn.CONFIGS["llama3-8b-gqa"], layers=1, ctx=(8, 8), vocab=5000), 31)
    logits = torch.tensor(syn.widen(w.logits, "bf16")).to(torch.bfloat16).cuda()
    idx = torch.empty((w.n_total, 4), dtype=torch.int32, device="cuda")
    val = torch.empty((w.n_total, 4), dtype=torch.float32, device="cuda")
    ptd.topk_draft(logits, 4, idx, val)
    drafts = [idx.cpu().numpy()]
    forests = [(list(map(int, w.trees[0])), list(map(int, w.tokens[:w.n_total])))]
    for expand in (1, 2):
        got, status, stride = _run(forests, drafts, expand, 4, 6, 128, dstride=4)
        assert status == 0
        _check(got, forests, drafts, expand, 4, 6, 128, stride)


def test_deep_chain_and_full_capacity():
    g = np.random.default_rng(7)
    chain = ([-1] + list(range(127)), list(range(128)))
    drafts = [g.integers(0, 500, size=(128, 2))]
    for max_depth in (1, 64, 127, 128):
        got, status, stride = _run([chain], drafts, 1, 2, max_depth, 128)
        assert status == 0      # full: nothing can be added; a depth above max_depth is stepped once
        _check(got, [chain], drafts, 1, 2, max_depth, 128, stride)
    short = ([-1] + list(range(99)), list(range(100)))
    got, status, stride = _run([short], [g.integers(0, 500, size=(100, 2))], 2, 3, 200, 128)
    assert status == 0 and got["count"][0] == 128   # additions stop at the capacity


def test_empty_and_invalid_forests():
    g = np.random.default_rng(8)
    good = _forest(g, 20, 6)
    bad = (list(good[0]), list(good[1]))
    bad[0][5] = 9                                   # a parent after its child
    forests = [good, ([], []), bad, good]
    drafts = [g.integers(0, 6, size=(20, 2)), np.zeros((1, 2), np.int64), g.integers(0, 6, size=(20, 2)),
              g.integers(0, 6, size=(20, 2))]
    got, status, stride = _run(forests, drafts, 2, 3, 4, 64)
    assert status == ptd.INVALID_TREE
    assert got["count"][2] == 0 and (got["parents"][2] == -1).all() and (got["o2n"][2] == -1).all()
    _check(got, [forests[0]], [drafts[0]], 2, 3, 4, 64, stride)
    assert got["count"][1] == 0 and (got["parents"][1] == -1).all()
    g3 = {k: v[3:4] for k, v in got.items()}
    _check(g3, [forests[3]], [drafts[3]], 2, 3, 4, 64, stride)


def test_chained_steps_on_device():
    """Ten steps in a row, each step's output forest (stride = capacity) fed back as the
    next input, against the oracle iterated on the host."""
    g = np.random.default_rng(9)
    B, cap = 3, 96
    host = [_forest(g, int(g.integers(1, 30)), 10) for _ in range(B)]
    cnt = torch.tensor([len(p) for p, _ in host], dtype=torch.int32, device="cuda")
    par = torch.full((B, cap), -1, dtype=torch.int32, device="cuda")
    tok = torch.full((B, cap), -1, dtype=torch.int32, device="cuda")
    for b, (p, t) in enumerate(host):
        par[b, :len(p)] = torch.tensor(p, dtype=torch.int32)
        tok[b, :len(t)] = torch.tensor(t, dtype=torch.int32)
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    for step in range(10):
        dr = g.integers(0, 10, size=(B * cap, 3))
        drafts = torch.tensor(dr, dtype=torch.int32, device="cuda")
        o = [torch.empty_like(x) for x in (cnt, par, tok, par, par)]
        ptd.draft_tree_update(cnt, par, tok, drafts, 2, 3, 5, cap, o[0], o[1], o[2], o[3], o[4], status)
        new_host = []
        for b, (p, t) in enumerate(host):
            want = oracle.draft_tree_update(p, t, dr[b * cap:b * cap + max(1, len(p))], 2, 3, 5, cap)
            new_host.append((want[0].tolist(), want[1].tolist()))
        cnt, par, tok = o[0], o[1], o[2]
        torch.cuda.synchronize()
        host = new_host
        for b, (p, t) in enumerate(host):
            assert int(cnt[b]) == len(p)
            assert par[b, :len(p)].tolist() == p and tok[b, :len(t)].tolist() == t
    assert int(status.item()) == 0
