"""Parity of the CUDA path (through the C ABI) with the CPU oracle.

Bit-exact: top-k indices and values, accepted paths / lengths / bonus tokens, compacted
cache bytes.  Attention: max-abs 2e-2 and mean-abs 2e-3 for bf16 inputs with fp32
accumulation, 1e-4 for fp32, plus a relative-RMS bound of 1e-2 and small / peaked
contexts, because at long contexts one wrongly (un)masked tree key moves an output by
only ~1/C (far below 2e-2).
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2607_10661_gb300 import ptd
from paper_2607_10661_gb300 import synthetic as syn
from paper_2607_10661_gb300.harness import DeviceWorkload, to_torch

pytestmark = pytest.mark.gpu

BF16_MAX, BF16_MEAN, REL_RMS = 2e-2, 2e-3, 1e-2
F32_MAX = 1e-4


@pytest.fixture(scope="module", autouse=True)
def _built():
    import __graft_entry__

    __graft_entry__.build()


def _attn_ref(w, layer, b, heads=None):
    """Oracle attention of tree b in one layer ([T, Hq, D]); optionally one KV group only."""
    c = w.cfg
    q = syn.widen(w.q_layer(layer), c.dtype)[w.nodes_of(b)]
    kc, vc = (syn.widen(x, c.dtype) for x in w.kv_layer(layer))
    k, v = w.seq_view(kc, b), w.seq_view(vc, b)
    if heads is not None:
        G = c.hq // c.hkv
        kvh = heads // G
        q = q[:, kvh * G:(kvh + 1) * G]
        k, v = k[:, kvh:kvh + 1], v[:, kvh:kvh + 1]
    return oracle.tree_attention(q, k, v, w.trees[b], int(w.ctx_lens[b]))


def _check_attn(got, ref, dtype, what=""):
    err = np.abs(got - ref)
    if dtype == "f32":
        assert err.max() <= F32_MAX, (what, err.max())
        return
    assert err.max() <= BF16_MAX, (what, err.max())
    assert err.mean() <= BF16_MEAN, (what, err.mean())
    rel = np.sqrt((err ** 2).mean() / max((ref ** 2).mean(), 1e-30))
    assert rel <= REL_RMS, (what, rel)


def _run_attention(w):
    dw = DeviceWorkload(w, with_step_buffers=False)
    dw.attention()
    torch.cuda.synchronize()
    assert int(dw.dev_status.item()) == 0
    return dw, dw.attn_out.float().cpu().numpy()


# ------------------------------------------------------------------------------ attention

ATTN_CASES = {
    # name: (base config, overrides) -- sizes the oracle finishes in seconds, spanning several
    # 128-key tiles, a ragged tail, one and two M tiles, units split between CTAs, fewer key
    # tiles than SMs, and the paged layout
    "tiny-fp32": ("tiny-fp32", {}),
    "fp32-d128-gqa": ("tiny-fp32", dict(hq=8, hkv=2, d=128, ctx=(300, 300))),
    "llama2-layer-short": ("llama2-7b-layer", dict(hq=8, hkv=8, ctx=(333, 333), vocab=100)),
    "llama3-gqa-2layers": ("llama3-8b-gqa", dict(layers=2, ctx=(1000, 1000), vocab=100)),
    "llama3-gqa-ctx0": ("llama3-8b-gqa", dict(layers=1, ctx=(0, 0), vocab=100)),
    "llama3-gqa-ctx1": ("llama3-8b-gqa", dict(layers=1, ctx=(1, 1), vocab=100)),
    "llama3-gqa-ctx7": ("llama3-8b-gqa", dict(layers=1, ctx=(7, 7), vocab=100)),
    "llama3-gqa-ctx65": ("llama3-8b-gqa", dict(layers=1, ctx=(65, 65), vocab=100)),
    "llama3-gqa-ctx128": ("llama3-8b-gqa", dict(layers=1, ctx=(128, 128), vocab=100)),
    "batched-paged-short": ("batched-paged", dict(ctx=(100, 700), vocab=100)),
    "long-context-short": ("long-context", dict(ctx=(3000, 3000), vocab=100)),
    "chain-128": ("llama3-8b-gqa", dict(layers=1, ctx=(50, 50), vocab=100, tree="chain", nodes=(128, 128))),
    "single-node": ("llama3-8b-gqa", dict(layers=1, ctx=(200, 200), vocab=100, tree="chain", nodes=(1, 1))),
    "mha-g1-t64": ("llama2-7b-layer", dict(hq=4, hkv=4, ctx=(129, 129), vocab=100, tree="chain",
                                           nodes=(64, 64))),
    # 18 key tiles on 18 CTAs, one each; the last tile starts at node 63 of a complete binary
    # tree, so within one warp nodes 88..94 first see a visible key (themselves) in chunk 0
    # and node 95 only in chunk 1: the lazy rescale must still run warp-uniformly
    "split-on-tree-tile": ("llama3-8b-gqa", dict(layers=1, hq=4, hkv=1, ctx=(961, 961), vocab=100, tree="binary",
                                                  nodes=(127, 127))),
}


@pytest.mark.parametrize("case", list(ATTN_CASES))
def test_attention_matches_oracle(case):
    base, over = ATTN_CASES[case]
    w = syn.Workload(syn.shrink(syn.CONFIGS[base], **over), 11)
    dw, got = _run_attention(w)
    for l in range(w.cfg.layers):
        for b in range(w.cfg.batch):
            ref = _attn_ref(w, l, b)
            _check_attn(got[l][w.nodes_of(b)], ref, w.cfg.dtype, f"{case} l{l} b{b}")


@pytest.mark.parametrize("case", ["llama3-gqa-2layers", "batched-paged-short", "split-on-tree-tile"])
def test_attention_without_workspace_matches_oracle(case):
    """No scratch: each (layer, tree, KV head, 256-row block) in one CTA, same results."""
    base, over = ATTN_CASES[case]
    w = syn.Workload(syn.shrink(syn.CONFIGS[base], **over), 11)
    dw = DeviceWorkload(w, with_step_buffers=False)
    dw.workspace = None
    dw.attention()
    torch.cuda.synchronize()
    assert int(dw.dev_status.item()) == 0
    got = dw.attn_out.float().cpu().numpy()
    for l in range(w.cfg.layers):
        for b in range(w.cfg.batch):
            _check_attn(got[l][w.nodes_of(b)], _attn_ref(w, l, b), w.cfg.dtype, f"{case} l{l} b{b}")


@pytest.mark.parametrize("layers,ctx,launches", [
    (12, 2000, 2),   # 96 units on 152 CTAs: pieces merged by the merge kernel, two column parts per unit
    (4, 2000, 2),    # 32 units: four column parts per unit
    (20, 1000, 1),   # 160 units: the last piece of each split unit merges inside the attention
])
def test_attention_merge_paths_match_oracle(layers, ctx, launches):
    """Both merges of split units (in the attention kernel, or by the merge kernel with two or
    four column parts per unit), every unit against the oracle."""
    cfg = syn.shrink(syn.CONFIGS["llama3-8b-gqa"], layers=layers, ctx=(ctx, ctx), vocab=100)
    w = syn.Workload(cfg, 23)
    dw = DeviceWorkload(w, with_step_buffers=False)
    n = dw.attention()
    torch.cuda.synchronize()
    assert int(dw.dev_status.item()) == 0
    if torch.cuda.get_device_properties(0).multi_processor_count == 152:
        assert n == launches
    got = dw.attn_out.float().cpu().numpy()
    for l in range(layers):
        _check_attn(got[l][w.nodes_of(0)], _attn_ref(w, l, 0), cfg.dtype, f"layers {layers} l{l}")


def test_attention_peaked_context_exposes_mask():
    """Committed-context keys made to score very low: outputs are dominated by the tree
    keys, so a wrongly (un)masked ancestor changes an output by O(1)."""
    cfg = syn.shrink(syn.CONFIGS["llama3-8b-gqa"], layers=1, ctx=(257, 257), vocab=100)
    w = syn.Workload(cfg, 5)
    dw = DeviceWorkload(w, with_step_buffers=False)
    C = int(w.ctx_lens[0])
    q = syn.widen(w.q_layer(0), "bf16")
    kc, vc = (syn.widen(x, "bf16") for x in w.kv_layer(0))
    # context keys = -4 * mean query direction of their group, so scores are strongly negative
    G = cfg.hq // cfg.hkv
    for h in range(cfg.hkv):
        dirn = q[:, h * G:(h + 1) * G].mean(axis=(0, 1))
        kc[0, :C, h] = -4.0 * dirn / np.linalg.norm(dirn) * np.sqrt(cfg.d)
    kbits = syn.bf16_bits(kc.astype(np.float32))
    dw.k[0].copy_(to_torch(kbits, "bf16"))
    kc = syn.widen(kbits, "bf16")
    dw.attention()
    torch.cuda.synchronize()
    ref = oracle.tree_attention(q, w.seq_view(kc, 0), w.seq_view(vc, 0), w.trees[0], C)
    got = dw.attn_out[0].float().cpu().numpy()
    _check_attn(got, ref, "bf16", "peaked")
    # and the tree part really dominates: dropping the ancestors changes the answer a lot
    flat = oracle.tree_attention(q, w.seq_view(kc, 0), w.seq_view(vc, 0), [-1] + [0] * (w.n_total - 1), C)
    assert np.abs(flat - ref).max() > 0.1


def _check_every_unit(w, got, what, layers=None):
    """Oracle attention of every (layer, tree, KV head) unit of a workload, each unit checked
    on its own (a per-unit tolerance, so that one wrong unit cannot hide in a mean over the
    others).  `got` is the kernel's [L][N_tot][Hq][D] output."""
    c = w.cfg
    G = c.hq // c.hkv
    for l in (range(c.layers) if layers is None else layers):
        q_all = syn.widen(w.q_layer(l), c.dtype)
        kc, vc = (syn.widen(x, c.dtype) for x in w.kv_layer(l))
        for b in range(c.batch):
            sl = w.nodes_of(b)
            ref = oracle.tree_attention(q_all[sl], w.seq_view(kc, b), w.seq_view(vc, b), w.trees[b],
                                        int(w.ctx_lens[b]))
            for kvh in range(c.hkv):
                hs = slice(kvh * G, (kvh + 1) * G)
                _check_attn(got[l][sl][:, hs], ref[:, hs], c.dtype, f"{what} l{l} b{b} kv{kvh}")


def test_attention_full_size_llama2_layer():
    """The Llama-2-7B-shaped layer at its own size: 32 MHA heads (M = 31 rows per unit, one
    128-row tcgen05 tile mostly padding), context 2048 (17 key tiles), every head."""
    w = syn.Workload(syn.CONFIGS["llama2-7b-layer"], 2000)
    assert (w.cfg.hq, w.cfg.hkv, int(w.ctx_lens[0]), w.n_total) == (32, 32, 2048, 31)
    dw, got = _run_attention(w)
    _check_every_unit(w, got, "llama2")


def test_attention_full_size_llama3_every_unit():
    """32 layers, context 8192, 63 nodes, the launch the benchmark times: all 256 (layer, KV
    head) units against the oracle.  With 152 persistent CTAs over 256 x 65 key tiles most
    units are cut between two CTAs and finished by the merge of their pieces."""
    w = syn.Workload(syn.CONFIGS["llama3-8b-gqa"], 1000)
    dw, got = _run_attention(w)
    _check_every_unit(w, got, "llama3")


def test_attention_full_size_long_context_every_head():
    """Context 32768, 128 nodes, 64 query / 8 KV heads: every KV head (each unit spans
    several CTAs' ranges)."""
    w = syn.Workload(syn.CONFIGS["long-context"], 5000)
    dw, got = _run_attention(w)
    _check_every_unit(w, got, "long")


def test_attention_full_size_batched_paged_every_unit():
    """Eight ragged sequences over a paged cache: every sequence and every KV head."""
    w = syn.Workload(syn.CONFIGS["batched-paged"], 4000)
    dw, got = _run_attention(w)
    _check_every_unit(w, got, "paged")


def test_attention_is_bit_reproducible():
    """Two launches on the same inputs write the same bits: the merge of a unit's pieces runs
    in a fixed order whatever piece finishes last."""
    w = syn.Workload(syn.shrink(syn.CONFIGS["long-context"], ctx=(6000, 6000), vocab=100), 17)
    dw = DeviceWorkload(w, with_step_buffers=False)
    outs = []
    for _ in range(3):
        dw.attn_out.zero_()
        dw.attention()
        torch.cuda.synchronize()
        outs.append(dw.attn_out.clone())
    assert int(dw.dev_status.item()) == 0
    assert torch.equal(outs[0], outs[1]) and torch.equal(outs[0], outs[2])


def test_attention_invalid_tree_reports_and_zeroes():
    cfg = syn.shrink(syn.CONFIGS["llama3-8b-gqa"], layers=1, ctx=(100, 100), vocab=100)
    w = syn.Workload(cfg, 2)
    dw = DeviceWorkload(w, with_step_buffers=False)
    bad = w.parents.copy()
    bad[5] = 7                                  # parent after the child
    dw.parents.copy_(torch.tensor(bad))
    dw.attn_out.fill_(1.0)
    dw.attention()
    torch.cuda.synchronize()
    assert int(dw.dev_status.item()) == ptd.INVALID_TREE
    assert float(dw.attn_out.abs().max()) == 0.0


# ------------------------------------------------------------------------------ top-k

@pytest.mark.parametrize("name", syn.CONFIG_ORDER)
def test_topk_matches_oracle(name):
    w = syn.Workload(syn.CONFIGS[name], 21)
    dev = torch.device("cuda:0")
    logits = to_torch(w.logits, w.cfg.dtype).to(dev)
    k = w.cfg.k
    idx = torch.zeros((w.n_total, k), dtype=torch.int32, device=dev)
    val = torch.zeros((w.n_total, k), dtype=torch.float32, device=dev)
    ptd.topk_draft(logits, k, idx, val)
    torch.cuda.synchronize()
    ref_i, ref_v = oracle.topk_rows(syn.widen(w.logits, w.cfg.dtype), k)
    assert np.array_equal(idx.cpu().numpy(), ref_i)
    assert np.array_equal(val.cpu().numpy().astype(np.float64), ref_v)


@pytest.mark.parametrize("dtype", ["bf16", "f32"])
@pytest.mark.parametrize("vocab,k", [(1, 1), (7, 3), (9, 9), (1001, 16), (32003, 5), (128256, 1), (152067, 16)])
def test_topk_edge_cases(dtype, vocab, k):
    g = np.random.default_rng(vocab + k)
    rows = 37
    x = np.round(g.standard_normal((rows, vocab)) * 2, 1).astype(np.float32)   # many ties
    x[:, ::5] = 0.0
    x[:, 3::7] = -0.0
    x[0] = 1.5                                                                 # a constant row
    if dtype == "bf16":
        bits = syn.bf16_bits(x)
        host, wide = bits, syn.widen(bits, "bf16")
    else:
        host, wide = x, x.astype(np.float64)
    # row stride not a multiple of 8 elements: rows start at every alignment
    stride = vocab + 3
    pad = np.zeros((rows, stride), dtype=host.dtype)
    pad[:, :vocab] = host
    t = to_torch(pad, dtype).cuda()
    idx = torch.zeros((rows, k), dtype=torch.int32, device="cuda")
    val = torch.zeros((rows, k), dtype=torch.float32, device="cuda")
    st = ptd.lib().ptd_topk_draft(t.data_ptr(), ptd.BF16 if dtype == "bf16" else ptd.F32, rows, vocab, stride, k,
                                  idx.data_ptr(), val.data_ptr(), torch.cuda.current_stream().cuda_stream)
    assert st == ptd.OK
    torch.cuda.synchronize()
    ref_i, ref_v = oracle.topk_rows(wide, k)
    assert np.array_equal(idx.cpu().numpy(), ref_i)
    assert np.array_equal(val.cpu().numpy().astype(np.float64), ref_v)


def test_topk_rejects_bad_k():
    t = torch.zeros((2, 10), dtype=torch.bfloat16, device="cuda")
    idx = torch.zeros((2, 17), dtype=torch.int32, device="cuda")
    val = torch.zeros((2, 17), dtype=torch.float32, device="cuda")
    with pytest.raises(ptd.PtdError):
        ptd.topk_draft(t, 17, idx, val)
    with pytest.raises(ptd.PtdError):
        ptd.topk_draft(t, 11, idx, val)


# ------------------------------------------------------------------------------ verify

def _verify_gpu(trees, tokens, target, max_nodes=None):
    dev = "cuda"
    offs = np.zeros(len(trees) + 1, np.int32)
    offs[1:] = np.cumsum([len(t) for t in trees])
    max_nodes = max_nodes or max(len(t) for t in trees)
    tree = ptd.Tree(torch.tensor(offs, device=dev), torch.tensor(np.concatenate(trees).astype(np.int32), device=dev),
                    torch.zeros(len(trees), dtype=torch.int32, device=dev), max_nodes, 0)
    B = len(trees)
    acc = torch.full((B, max_nodes), 77, dtype=torch.int32, device=dev)
    alen = torch.zeros(B, dtype=torch.int32, device=dev)
    bonus = torch.zeros(B, dtype=torch.int32, device=dev)
    st = torch.zeros(1, dtype=torch.int32, device=dev)
    ptd.verify_greedy(tree, torch.tensor(tokens, dtype=torch.int32, device=dev),
                      torch.tensor(target, dtype=torch.int32, device=dev), 1, acc, alen, bonus, st)
    torch.cuda.synchronize()
    return acc.cpu().numpy(), alen.cpu().numpy(), bonus.cpu().numpy(), int(st.item())


def _expect_verify(trees, tokens, target, acc, alen, bonus):
    off = 0
    for b, par in enumerate(trees):
        T = len(par)
        path, n, bo = oracle.verify_greedy(par, tokens[off:off + T], target[off:off + T])
        assert alen[b] == n and bonus[b] == bo, (b, n, alen[b])
        assert acc[b, :n].tolist() == path
        assert (acc[b, n:] == -1).all()
        off += T


@pytest.mark.parametrize("name", syn.CONFIG_ORDER)
def test_verify_on_workloads(name):
    cfg = syn.CONFIGS[name]
    w = syn.Workload(syn.shrink(cfg, vocab=min(cfg.vocab, 3000)), 31)
    idx, _ = oracle.topk_rows(syn.widen(w.logits, w.cfg.dtype), 1)
    acc, alen, bonus, st = _verify_gpu(w.trees, w.tokens, idx[:, 0], w.max_nodes)
    assert st == 0
    _expect_verify(w.trees, w.tokens, idx[:, 0], acc, alen, bonus)


def test_verify_random_trees_dense_matches_and_ties():
    """Small alphabet: many eligible edges, duplicate sibling tokens (ties broken by the
    lexicographically smallest path), batch of ragged trees up to 128 nodes."""
    g = np.random.default_rng(3)
    for trial in range(20):
        trees, toks, tgts = [], [], []
        for b in range(int(g.integers(1, 9))):
            T = int(g.choice([1, 2, 3, 7, 31, 64, 127, 128]))
            par = np.array([-1] + [int(g.integers(max(0, i - 4), i)) for i in range(1, T)], np.int32)
            trees.append(par)
            toks.append(g.integers(0, 2, size=T))
            tgts.append(g.integers(0, 2, size=T))
        tokens, target = np.concatenate(toks).astype(np.int32), np.concatenate(tgts).astype(np.int32)
        acc, alen, bonus, st = _verify_gpu(trees, tokens, target)
        assert st == 0
        _expect_verify(trees, tokens, target, acc, alen, bonus)


def test_verify_full_chain_accepts_all_128():
    par = np.arange(-1, 127, dtype=np.int32)
    tokens = np.arange(128, dtype=np.int32)
    target = np.arange(1, 129, dtype=np.int32)      # V_n = token of node n+1
    acc, alen, bonus, st = _verify_gpu([par], tokens, target)
    assert st == 0 and alen[0] == 128 and bonus[0] == 128 and acc[0].tolist() == list(range(128))


def test_verify_invalid_tree():
    good = np.array([-1, 0, 0, 1], np.int32)
    bad = np.array([-1, 0, 3, 1], np.int32)
    acc, alen, bonus, st = _verify_gpu([good, bad], np.zeros(8, np.int32), np.zeros(8, np.int32))
    assert st == ptd.INVALID_TREE
    assert alen[1] == 0 and bonus[1] == -1 and (acc[1] == -1).all()
    assert alen[0] == 3   # the valid tree is still verified (all tokens and targets 0)


# ------------------------------------------------------------------------------ compaction

@pytest.mark.parametrize("name", ["llama3-8b-gqa", "batched-paged", "tiny-fp32"])
def test_compact_matches_oracle(name):
    cfg = syn.CONFIGS[name]
    over = dict(vocab=min(cfg.vocab, 2000))
    if name == "llama3-8b-gqa":
        over.update(layers=3, ctx=(300, 300))
    w = syn.Workload(syn.shrink(cfg, **over), 41)
    cfg = w.cfg
    dw = DeviceWorkload(w, with_step_buffers=False)
    # a chosen root path per tree: the deepest node's ancestors (long, overlapping copies)
    B, M = cfg.batch, w.max_nodes
    acc = np.full((B, M), -1, np.int32)
    alen = np.zeros(B, np.int32)
    for b, par in enumerate(w.trees):
        d = oracle.depths(par)
        end = int(np.argmax(d))
        path = [end]
        while par[path[-1]] >= 0:
            path.append(int(par[path[-1]]))
        path.reverse()
        acc[b, :len(path)] = path
        alen[b] = len(path)
    k_before, v_before = dw.k.cpu(), dw.v.cpu()
    dw.accepted.copy_(torch.tensor(acc))
    dw.accept_len.copy_(torch.tensor(alen))
    dw.compact()
    torch.cuda.synchronize()
    k_after, v_after = dw.k.cpu(), dw.v.cpu()
    assert dw.new_ctx.cpu().numpy().tolist() == (w.ctx_lens + alen).tolist()
    for before, after in ((k_before, k_after), (v_before, v_after)):
        bb = before.view(torch.int16).numpy() if before.dtype == torch.bfloat16 else before.numpy()
        aa = after.view(torch.int16).numpy() if after.dtype == torch.bfloat16 else after.numpy()
        for l in range(cfg.layers):
            for b in range(B):
                C = int(w.ctx_lens[b])
                n = int(alen[b])
                seq_b = w.seq_view(bb[l], b)
                seq_a = w.seq_view(aa[l], b)
                ref, new_ctx = oracle.kv_compact(seq_b, acc[b, :n], C)
                assert np.array_equal(seq_a[:new_ctx], ref[:new_ctx])


@pytest.mark.parametrize("name", ["llama3-8b-gqa", "batched-paged", "tiny-fp32"])
def test_verify_and_compact_equals_the_two_calls(name):
    """ptd_verify_and_compact (one launch) leaves exactly what ptd_verify_greedy followed by
    ptd_kv_compact leave: path, length, bonus, status, new context and cache bytes; also with
    one tree made invalid."""
    cfg = syn.CONFIGS[name]
    over = dict(vocab=min(cfg.vocab, 64))
    if name == "llama3-8b-gqa":
        over.update(layers=3, ctx=(300, 300))
    outs = []
    for fused in (False, True):
        w = syn.Workload(syn.shrink(cfg, **over), 43)
        dw = DeviceWorkload(w)
        target = np.random.default_rng(7).integers(0, w.cfg.vocab, size=(w.n_total, w.cfg.k)).astype(np.int32)
        tokens = w.tokens.copy()
        for b, par in enumerate(w.trees):   # most edges eligible: deep, tied paths
            o = int(w.node_offsets[b])
            for i in range(1, len(par)):
                if (i * 7 + b) % 5:
                    tokens[o + i] = target[o + par[i], 0]
        bad = w.parents.copy()
        if w.cfg.batch > 1:
            o1 = int(w.node_offsets[1])
            bad[o1 + 2] = 5                   # tree 1: a parent after its child
        dw.parents.copy_(torch.tensor(bad))
        dw.tokens.copy_(torch.tensor(tokens))
        dw.topk_idx.copy_(torch.tensor(target))
        dw.dev_status.zero_()
        if fused:
            assert dw.verify_and_compact() == 1
        else:
            dw.verify()
            dw.compact()
        torch.cuda.synchronize()
        kk = dw.k.cpu()
        kk = kk.view(torch.int16) if kk.dtype == torch.bfloat16 else kk.view(torch.int32)
        outs.append((dw.accepted.cpu(), dw.accept_len.cpu(), dw.bonus.cpu(), dw.new_ctx.cpu(),
                     int(dw.dev_status.item()), kk))
    for x, y in zip(outs[0], outs[1]):
        if isinstance(x, int):
            assert x == y
        else:
            assert torch.equal(x, y)
    assert int(outs[0][1].max()) > 2


# ------------------------------------------------------------------------------ whole step

@pytest.mark.parametrize("case", ["tiny-fp32", "llama3-gqa-2layers", "batched-paged-short"])
def test_whole_step_matches_oracle(case):
    base, over = ATTN_CASES[case]
    cfg = syn.shrink(syn.CONFIGS[base], **over)
    w = syn.Workload(cfg, 51)
    dw = DeviceWorkload(w)
    k_before = dw.k.cpu()
    n_attn = dw.attention()                          # 1, or 2 with the merge of split units
    dw.attn_out.zero_()
    n = dw.step()
    assert n == n_attn + 2                           # attention, top-k, verify + compact
    torch.cuda.synchronize()
    assert int(dw.dev_status.item()) == 0
    got = dw.attn_out.float().cpu().numpy()
    for b in range(cfg.batch):
        _check_attn(got[0][w.nodes_of(b)], _attn_ref(w, 0, b), cfg.dtype, f"step b{b}")
    idx_ref, _ = oracle.topk_rows(syn.widen(w.logits, cfg.dtype), cfg.k)
    assert np.array_equal(dw.topk_idx.cpu().numpy(), idx_ref)
    kb = k_before.view(torch.int16).numpy() if k_before.dtype == torch.bfloat16 else k_before.numpy()
    ka = dw.k.cpu()
    ka = ka.view(torch.int16).numpy() if ka.dtype == torch.bfloat16 else ka.numpy()
    for b, par in enumerate(w.trees):
        sl = w.nodes_of(b)
        path, nacc, bonus = oracle.verify_greedy(par, w.tokens[sl], idx_ref[sl, 0])
        assert int(dw.accept_len[b]) == nacc and int(dw.bonus[b]) == bonus
        assert dw.accepted[b, :nacc].cpu().tolist() == path
        ref, new_ctx = oracle.kv_compact(w.seq_view(kb[0], b), path, int(w.ctx_lens[b]))
        assert int(dw.new_ctx[b]) == new_ctx
        assert np.array_equal(w.seq_view(ka[0], b)[:new_ctx], ref[:new_ctx])


@pytest.mark.parametrize("base,tree,seed", [("llama3-8b-gqa", "binary", 3), ("llama3-8b-gqa", "branching", 5),
                                            ("llama3-8b-gqa", "chain", 6), ("batched-paged", "random-depth", 4)])
def test_step_verify_compact_on_eligible_trees(base, tree, seed):
    """The step's fused verification + compaction on trees where most edges are eligible
    (draft token = the parent's greedy token) and several paths tie in depth, so the
    lexicographic choice and the compaction of a long path are exercised."""
    over = dict(layers=2, ctx=(150, 150), vocab=64, tree=tree)
    if tree in ("binary", "chain"):
        over["nodes"] = (63, 63)
    if base == "batched-paged":
        over.update(batch=2, hq=8, hkv=2)
    cfg = syn.shrink(syn.CONFIGS[base], **over)
    w = syn.Workload(cfg, seed)
    dw = DeviceWorkload(w)
    idx_ref, _ = oracle.topk_rows(syn.widen(w.logits, cfg.dtype), cfg.k)
    greedy = idx_ref[:, 0]
    rng = np.random.default_rng(seed)
    tokens = w.tokens.copy()
    for b, par in enumerate(w.trees):
        o = int(w.node_offsets[b])
        for i in range(1, len(par)):
            tokens[o + i] = greedy[o + par[i]] if rng.random() < 0.8 else int(rng.integers(cfg.vocab))
    dw.tokens.copy_(torch.tensor(tokens, dtype=torch.int32))
    k_before = dw.k.cpu().view(torch.int16).numpy()
    assert dw.step() in (3, 4)   # attention (+ the merge of split units), top-k (+ verification), compaction
    torch.cuda.synchronize()
    assert int(dw.dev_status.item()) == 0
    ka = dw.k.cpu().view(torch.int16).numpy()
    for b, par in enumerate(w.trees):
        sl = w.nodes_of(b)
        path, nacc, bonus = oracle.verify_greedy(par, tokens[sl], greedy[sl])
        assert nacc > 2
        assert int(dw.accept_len[b]) == nacc and int(dw.bonus[b]) == bonus
        acc = dw.accepted[b].cpu().tolist()
        assert acc[:nacc] == path and all(x == -1 for x in acc[nacc:])
        for l in range(cfg.layers):
            ref, new_ctx = oracle.kv_compact(w.seq_view(k_before[l], b), path, int(w.ctx_lens[b]))
            assert int(dw.new_ctx[b]) == new_ctx
            assert np.array_equal(w.seq_view(ka[l], b)[:new_ctx], ref[:new_ctx])


def test_full_size_step_compaction_after_attention():
    """The one-call step at the benchmark's size (32 layers, context 8192, 63 nodes, vocab
    128256), with draft tokens made mostly eligible so the accepted path leaves the first
    children and the compaction overwrites tree slots that the attention reads.  The top-k of
    this entry starts while the attention grid drains and the compaction waits on the top-k
    grid only: every sampled attention output must still match the oracle on the cache as it
    was before the step, and every layer's cache must hold the compacted path."""
    w = syn.Workload(syn.CONFIGS["llama3-8b-gqa"], 1001)
    cfg = w.cfg
    dw = DeviceWorkload(w)
    idx_ref, _ = oracle.topk_rows(syn.widen(w.logits, cfg.dtype), cfg.k)
    greedy = idx_ref[:, 0]
    par = w.trees[0]
    rng = np.random.default_rng(7)
    tokens = w.tokens.copy()
    # eligible everywhere except the first child of the root, so the path leaves node 1
    first_child = min(i for i in range(1, len(par)) if par[i] == 0)
    for i in range(1, len(par)):
        tokens[i] = greedy[par[i]] if (i != first_child and rng.random() < 0.9) else (greedy[par[i]] + 1) % cfg.vocab
    dw.tokens.copy_(torch.tensor(tokens, dtype=torch.int32))
    path, nacc, bonus = oracle.verify_greedy(par, tokens, greedy)
    assert nacc > 2 and any(path[j] != j for j in range(nacc))
    k_before = dw.k.cpu().view(torch.int16).numpy()
    assert dw.step() in (3, 4)   # attention (+ the merge of split units), top-k (+ verification), compaction
    torch.cuda.synchronize()
    assert int(dw.dev_status.item()) == 0
    assert int(dw.accept_len[0]) == nacc and int(dw.bonus[0]) == bonus
    assert dw.accepted[0, :nacc].cpu().tolist() == path
    got = dw.attn_out.float().cpu().numpy()
    _check_every_unit(w, got, "step", layers=range(0, cfg.layers, 3))
    ka = dw.k.cpu().view(torch.int16).numpy()
    for l in range(cfg.layers):
        ref, new_ctx = oracle.kv_compact(w.seq_view(k_before[l], 0), path, int(w.ctx_lens[0]))
        assert int(dw.new_ctx[0]) == new_ctx
        assert np.array_equal(w.seq_view(ka[l], 0)[:new_ctx], ref[:new_ctx])


def test_host_step_matches_device_step():
    """ptd_tree_verify_step_host (pinned host inputs and outputs) gives the device step's results."""
    cfg = syn.shrink(syn.CONFIGS["llama3-8b-gqa"], layers=2, ctx=(700, 700), vocab=3000)
    w = syn.Workload(cfg, 61)
    dw = DeviceWorkload(w)
    n_attn = dw.attention()                          # 1, or 2 with the merge of split units
    N, L = w.n_total, cfg.layers
    C = int(w.ctx_lens[0])
    pin = lambda t: t.contiguous().pin_memory()
    tree_k = pin(torch.stack([dw.k[l, 0, C:C + N] for l in range(L)]).cpu())
    tree_v = pin(torch.stack([dw.v[l, 0, C:C + N] for l in range(L)]).cpu())
    io_t = dict(q_h=pin(dw.q.cpu()), logits_h=pin(dw.logits.cpu()), tokens_h=pin(dw.tokens.cpu()),
                parents_h=pin(dw.parents.cpu()), node_offsets_h=pin(dw.node_offsets.cpu()),
                ctx_lens_h=pin(dw.ctx_lens.cpu()), tree_k_h=tree_k, tree_v_h=tree_v,
                topk_idx_h=pin(torch.zeros((N, cfg.k), dtype=torch.int32)),
                topk_val_h=pin(torch.zeros((N, cfg.k), dtype=torch.float32)),
                accepted_h=pin(torch.zeros((1, w.max_nodes), dtype=torch.int32)),
                accept_len_h=pin(torch.zeros(1, dtype=torch.int32)), bonus_h=pin(torch.zeros(1, dtype=torch.int32)),
                new_ctx_h=pin(torch.zeros(1, dtype=torch.int32)), status_h=pin(torch.zeros(1, dtype=torch.int32)))
    io = ptd.HostIO(**io_t)
    # scramble the device inputs: the host call must overwrite them
    dw.q.zero_()
    dw.logits.zero_()
    n = ptd.tree_verify_step_host(dw.tree, dw.cache, dw.bufs, io)
    assert n == n_attn + 2                           # attention, top-k, verify + compact
    torch.cuda.synchronize()
    idx_ref, _ = oracle.topk_rows(syn.widen(w.logits, cfg.dtype), cfg.k)
    assert np.array_equal(io_t["topk_idx_h"].numpy(), idx_ref)
    path, nacc, bonus = oracle.verify_greedy(w.trees[0], w.tokens, idx_ref[:, 0])
    assert int(io_t["accept_len_h"][0]) == nacc and int(io_t["bonus_h"][0]) == bonus
    assert io_t["accepted_h"][0, :nacc].tolist() == path
    assert int(io_t["new_ctx_h"][0]) == C + nacc and int(io_t["status_h"][0]) == 0
    got = dw.attn_out.float().cpu().numpy()
    _check_attn(got[1], _attn_ref(w, 1, 0), "bf16", "host step")


# ------------------------------------------------------------------------------ sampling verification

SAMPLING_CASES = {
    # name: (base config, overrides, temperature[, workload seed])
    "llama3-full-vocab-peaked": ("llama3-8b-gqa", dict(layers=1, ctx=(8, 8)), 0.1),
    "llama3-full-vocab-flat": ("llama3-8b-gqa", dict(layers=1, ctx=(8, 8)), 1.0),
    "batched-3-trees": ("batched-paged", dict(batch=3, layers=1, ctx=(16, 32), vocab=32000, hq=8, hkv=2), 0.5),
    "tiny-fp32": ("tiny-fp32", {}, 0.8),
    "single-node": ("llama3-8b-gqa", dict(layers=1, ctx=(8, 8), vocab=5000, tree="chain", nodes=(1, 1)), 1.0),
    # a 4-CTA cluster, and rows that are not 16-byte aligned (scalar loads)
    "odd-vocab-50001": ("llama3-8b-gqa", dict(layers=1, ctx=(8, 8), vocab=50001), 0.7),
    # fp32 logits over a 5-CTA cluster with vector loads
    "fp32-vocab-70000": ("tiny-fp32", dict(vocab=70000), 1.0),
    # chunks longer than 32 logits (the kernel reads them from memory in pieces)
    "vocab-200000": ("llama3-8b-gqa", dict(layers=1, ctx=(8, 8), vocab=200000), 1.0),
    # acceptance uniforms in [0.5, 1) and a root row whose top token has P ~0.75 (workload
    # seed 77): a child carrying it is rejected, leaving a small residual for its siblings
    # and the bonus
    "llama3-dominant-rejected": ("llama3-8b-gqa", dict(layers=1, ctx=(8, 8)), 0.2, 77),
}
MARGIN = 2e-6   # fp32 exponentials vs the oracle's float64: keep every decision this far from flipping


def _sampling_inputs(w, temp, seed, u_scale=1.0, u_lo=0.0):
    """Tokens that are mostly the parent's argmax (long accepted paths at low temperature)
    and uniforms whose every decision is at least MARGIN from its threshold."""
    cfg = w.cfg
    logits = syn.widen(w.logits, cfg.dtype)
    arg = logits.argmax(axis=1)
    g = np.random.default_rng(seed)
    tokens = w.tokens.copy()
    for b, par in enumerate(w.trees):
        o = int(w.node_offsets[b])
        for i in range(1, len(par)):
            tokens[o + i] = arg[o + par[i]] if g.random() < 0.6 else int(g.integers(cfg.vocab))
    u_acc = np.zeros(w.n_total, np.float32)
    u_bon = np.zeros(cfg.batch, np.float32)
    refs = []
    for b, par in enumerate(w.trees):
        sl = w.nodes_of(b)
        for _ in range(200):
            ua = (u_lo + g.random(len(par)) * (u_scale - u_lo)).astype(np.float32)
            ub = np.float32(g.random())
            ref = oracle.verify_sampling(par, tokens[sl], logits[sl], temp, ua.astype(np.float64), float(ub))
            if ref[3] > MARGIN:
                break
        assert ref[3] > MARGIN
        u_acc[sl] = ua
        u_bon[b] = ub
        refs.append(ref)
    return tokens, u_acc, u_bon, refs


def _run_sampling_case(case, pad=None):
    base, over, temp, *seed = SAMPLING_CASES[case]
    w = syn.Workload(syn.shrink(syn.CONFIGS[base], **over), seed[0] if seed else 71)
    dw = DeviceWorkload(w)
    # peaked: acceptance uniforms in [0, 0.05) accept every child carrying its parent's argmax
    for seed in range(72, 122):
        tokens, u_acc, u_bon, refs = _sampling_inputs(w, temp, seed, 0.05 if case.endswith("peaked") else 1.0,
                                                      0.5 if case.endswith("rejected") else 0.0)
        # the dominant-rejected case takes the first draw that rejects a dominant token
        if not case.endswith("rejected") or _max_rejected_p(w, tokens, temp, refs) > 0.5:
            break
    dw.tokens.copy_(torch.tensor(tokens, dtype=torch.int32))
    dw.dev_status.zero_()
    ua, ub = torch.tensor(u_acc, device="cuda"), torch.tensor(u_bon, device="cuda")
    logits = dw.logits
    if pad is not None:   # rows `pad` elements longer than the vocabulary, padding poisoned
        wide = torch.full((logits.shape[0], logits.shape[1] + pad), 1e4, dtype=logits.dtype, device=logits.device)
        wide[:, :logits.shape[1]] = logits
        logits = wide[:, :logits.shape[1]]
        assert logits.stride(0) == dw.logits.shape[1] + pad
    assert ptd.verify_sampling(dw.tree, dw.tokens, logits, temp, ua, ub, dw.accepted, dw.accept_len, dw.bonus,
                               dw.dev_status) == 1
    torch.cuda.synchronize()
    assert int(dw.dev_status.item()) == 0
    acc = dw.accepted.cpu().numpy()
    for b, (path, alen, bonus, _) in enumerate(refs):
        assert int(dw.accept_len[b]) == alen, (case, b)
        assert acc[b, :alen].tolist() == path and (acc[b, alen:] == -1).all()
        assert int(dw.bonus[b]) == bonus, (case, b)
    return w, tokens, temp, refs


def _max_rejected_p(w, tokens, temp, refs):
    """Largest P_v(token) among the children rejected along the oracle's decisions."""
    logits = syn.widen(w.logits, w.cfg.dtype)
    best = 0.0
    for b, par in enumerate(w.trees):
        o = int(w.node_offsets[b])
        path = refs[b][0]
        for i, v in enumerate(path):
            P = oracle.softmax_row(logits[o + v], temp)
            nxt = path[i + 1] if i + 1 < len(path) else None
            for n in range(v + 1, len(par)):
                if par[n] != v:
                    continue
                if n == nxt:
                    break
                best = max(best, float(P[int(tokens[o + n])]))
    return best


@pytest.mark.parametrize("case", list(SAMPLING_CASES))
def test_verify_sampling_matches_oracle(case):
    w, tokens, temp, refs = _run_sampling_case(case)
    if case == "llama3-full-vocab-peaked":
        assert max(r[1] for r in refs) >= 3     # long accepted paths are exercised
    if case == "llama3-dominant-rejected":
        assert _max_rejected_p(w, tokens, temp, refs) > 0.5   # a dominant token was rejected


@pytest.mark.parametrize("pad", [8, 3])
def test_verify_sampling_strided_rows(pad):
    """Rows further apart than the vocabulary: with a pad of 8 they stay 16-byte aligned
    (vector loads), with 3 they do not (scalar loads); the padding is never read."""
    _run_sampling_case("llama3-full-vocab-flat", pad)


def test_verify_sampling_invalid_tree_and_argument_checks():
    w = syn.Workload(syn.shrink(syn.CONFIGS["batched-paged"], batch=2, layers=1, ctx=(16, 16), vocab=1000, hq=8,
                                hkv=2), 73)
    dw = DeviceWorkload(w)
    bad = w.parents.copy()
    bad[int(w.node_offsets[1]) + 3] = 7            # tree 1: a parent after its child
    dw.parents.copy_(torch.tensor(bad))
    dw.dev_status.zero_()
    ua = torch.rand(w.n_total, device="cuda")
    ub = torch.rand(2, device="cuda")
    ptd.verify_sampling(dw.tree, dw.tokens, dw.logits, 1.0, ua, ub, dw.accepted, dw.accept_len, dw.bonus,
                        dw.dev_status)
    torch.cuda.synchronize()
    assert int(dw.dev_status.item()) == ptd.INVALID_TREE
    assert int(dw.accept_len[1]) == 0 and int(dw.bonus[1]) == -1 and (dw.accepted[1] == -1).all()
    assert int(dw.accept_len[0]) >= 1                # the valid tree is still verified
    with pytest.raises(RuntimeError):
        ptd.verify_sampling(dw.tree, dw.tokens, dw.logits, 0.0, ua, ub, dw.accepted, dw.accept_len, dw.bonus,
                            dw.dev_status)


# ------------------------------------------------------------------ the step's two tails

def _step_outputs(dw):
    kk = dw.k.cpu()
    kk = kk.view(torch.int16) if kk.dtype == torch.bfloat16 else kk.view(torch.int32)
    vv = dw.v.cpu()
    vv = vv.view(torch.int16) if vv.dtype == torch.bfloat16 else vv.view(torch.int32)
    return dict(idx=dw.topk_idx.cpu(), val=dw.topk_val.cpu(), acc=dw.accepted.cpu(), alen=dw.accept_len.cpu(),
                bonus=dw.bonus.cpu(), new_ctx=dw.new_ctx.cpu(), status=int(dw.dev_status.item()), k=kk, v=vv,
                out=dw.attn_out.cpu())


@pytest.mark.parametrize("base,over,seed", [
    ("llama3-8b-gqa", dict(layers=2, ctx=(300, 300), vocab=50000), 81),
    ("batched-paged", dict(ctx=(64, 400), vocab=3000), 82),
    # forty ragged trees of 1-16 nodes: several clusters finish rows of the same tree at once
    ("batched-paged", dict(batch=40, ctx=(16, 200), nodes=(1, 16), depth_range=(1, 4), vocab=700, hq=8, hkv=2), 83),
])
def test_step_fused_tail_equals_three_launch_tail(base, over, seed):
    """With the step's workspace (ptd_step_workspace_size) the top-k's CTAs verify the trees and
    a copy kernel compacts; with the attention's workspace alone the step runs the top-k and
    ptd_verify_and_compact (whose every CTA verifies its tree before copying).  Every output and the cache must be identical,
    on trees whose draft tokens mostly match their parent's greedy token (long tied paths), with
    one tree made invalid, and on two steps in a row (the counters' tags change per launch)."""
    cfg = syn.shrink(syn.CONFIGS[base], **over)
    outs = []
    for fused in (True, False):
        w = syn.Workload(cfg, seed)
        dw = DeviceWorkload(w)
        if not fused:
            small = ptd.attention_workspace_size(dw.tree, dw.cache, cfg.hq)
            ws = torch.empty(max(small, 16), dtype=torch.uint8, device="cuda")
            dw.bufs = ptd.StepBuffers(dw.q, cfg.hq, dw.attn_out, dw.logits, cfg.k, dw.tokens, dw.topk_idx,
                                      dw.topk_val, dw.accepted, dw.accept_len, dw.bonus, dw.new_ctx, dw.dev_status,
                                      ws if small else None)
        idx_ref, _ = oracle.topk_rows(syn.widen(w.logits, cfg.dtype), cfg.k)
        rng = np.random.default_rng(seed)
        tokens = w.tokens.copy()
        for b, par in enumerate(w.trees):
            o = int(w.node_offsets[b])
            for i in range(1, len(par)):
                tokens[o + i] = idx_ref[o + par[i], 0] if rng.random() < 0.85 else int(rng.integers(cfg.vocab))
        dw.tokens.copy_(torch.tensor(tokens, dtype=torch.int32))
        if cfg.batch > 2:
            bad = w.parents.copy()
            o = int(w.node_offsets[1])
            if int(w.node_offsets[2]) - o > 2:
                bad[o + 2] = 5 if int(w.node_offsets[2]) - o > 5 else -3    # tree 1: not a tree
                dw.parents.copy_(torch.tensor(bad))
        launches = []
        for _ in range(2):
            launches.append(dw.step())
        torch.cuda.synchronize()
        # attention (+ the merge of split units), top-k (+ verification), compaction
        assert launches[0] == launches[1] and launches[0] in (3, 4)
        outs.append(_step_outputs(dw))
        if cfg.batch <= 2:
            # and against the oracle: path, length and bonus of every tree
            for b, par in enumerate(w.trees):
                sl = w.nodes_of(b)
                path, n, bo = oracle.verify_greedy(par, tokens[sl], idx_ref[sl, 0])
                assert int(dw.accept_len[b]) == n and int(dw.bonus[b]) == bo
                assert dw.accepted[b, :n].cpu().tolist() == path
    a, b = outs
    for key in a:
        if isinstance(a[key], int):
            assert a[key] == b[key], key
        else:
            assert torch.equal(a[key], b[key]), key
    assert int(a["alen"].max()) > 2


# ------------------------------------------------------------------------------ streamed top-k of the step

# With the step's workspace and bf16 rows of a multiple of 8 logits, the step's top-k is the
# persistent streaming kernel: the rows back to back, one equal share per CTA, so a row is cut
# into parts that end in different CTAs and meet in a merge by the part that completes it.
STREAM_CASES = {
    # one row of 128256 logits in eight CTAs
    "one-row": ("llama3-8b-gqa", dict(layers=1, ctx=(64, 64), tree="chain", nodes=(1, 1)), 91),
    # three rows, CTA shares crossing the row boundaries
    "three-rows": ("llama3-8b-gqa", dict(layers=1, ctx=(64, 64), tree="chain", nodes=(3, 3)), 92),
    # forty trees of 1-16 nodes with 1000 logits a row: several rows in one CTA's share
    "many-short-rows": ("batched-paged", dict(batch=40, ctx=(16, 200), nodes=(1, 16), depth_range=(1, 4),
                                              vocab=1000, hq=8, hkv=2), 93),
    # 128 rows of 152064 logits, k = 6
    "long-context-rows": ("long-context", dict(layers=1, ctx=(200, 200)), 94),
    # eight trees of 16-64 nodes, 128256 logits a row (the batched workload's rows)
    "batched-rows": ("batched-paged", dict(ctx=(64, 300)), 97),
    # the largest k, and k = 1
    "k16": ("batched-paged", dict(batch=3, ctx=(64, 200), vocab=20000, k=16, hq=8, hkv=2), 95),
    "k1": ("llama3-8b-gqa", dict(layers=1, ctx=(64, 64), vocab=4096, k=1), 96),
}


def _plant_ties(w):
    """Every other row gets four equal maxima (one at each end, two adjacent in the middle,
    which straddle a CTA boundary in the one-row case); returns the bf16 bit patterns."""
    logits = w.logits.copy()
    f = syn.bf16_to_f32(logits)
    V = w.cfg.vocab
    cols = [5, V // 2 - 1, V // 2, V - 1]
    for r in range(0, logits.shape[0], 2):
        top = syn.bf16_bits(np.array([f[r].max() + 1.0], np.float32))[0]
        logits[r, cols] = top
    return logits


def _tree_counter_workspace(dw, cfg):
    """The attention's scratch and the per-tree counters only: the step's clustered top-k."""
    small = ptd.attention_workspace_size(dw.tree, dw.cache, cfg.hq)
    return (small + 255) // 256 * 256 + (4 * cfg.batch + 255) // 256 * 256


@pytest.mark.parametrize("case", list(STREAM_CASES))
def test_step_streamed_topk_matches_oracle(case):
    """Every top-k row (indices and values, ties to the lower index across CTA parts), every
    verified path and the compacted caches equal the oracle's, with the streamed top-k forced,
    with the clustered one forced, and with the clustered one chosen by a workspace that holds
    only the per-tree counters: identical outputs all three ways."""
    base, over, seed = STREAM_CASES[case]
    cfg = syn.shrink(syn.CONFIGS[base], **over)
    outs = []
    for kind in ("streamed", "clustered", "tree-counters"):
        w = syn.Workload(cfg, seed)
        dw = DeviceWorkload(w)
        logits = _plant_ties(w)
        dw.logits.copy_(to_torch(logits, cfg.dtype))
        if kind == "tree-counters":
            ws = torch.empty(_tree_counter_workspace(dw, cfg), dtype=torch.uint8, device="cuda")
            dw.bufs = ptd.StepBuffers(dw.q, cfg.hq, dw.attn_out, dw.logits, cfg.k, dw.tokens, dw.topk_idx,
                                      dw.topk_val, dw.accepted, dw.accept_len, dw.bonus, dw.new_ctx, dw.dev_status,
                                      ws)
        prev = ptd.step_topk_policy(ptd.STEP_TOPK_CLUSTERED if kind == "clustered" else ptd.STEP_TOPK_STREAMED)
        idx_ref, val_ref = oracle.topk_rows(syn.bf16_to_f32(logits), cfg.k)
        greedy = idx_ref[:, 0]
        rng = np.random.default_rng(seed)
        tokens = w.tokens.copy()
        for b, par in enumerate(w.trees):
            o = int(w.node_offsets[b])
            for i in range(1, len(par)):
                tokens[o + i] = greedy[o + par[i]] if rng.random() < 0.8 else int(rng.integers(cfg.vocab))
        dw.tokens.copy_(torch.tensor(tokens, dtype=torch.int32))
        k_before = dw.k.cpu().view(torch.int16).numpy()
        try:
            launches = dw.step()
            torch.cuda.synchronize()
        finally:
            ptd.step_topk_policy(prev)
        assert launches in (3, 4)
        assert int(dw.dev_status.item()) == 0
        assert np.array_equal(dw.topk_idx.cpu().numpy(), idx_ref)
        assert np.array_equal(dw.topk_val.cpu().numpy(), val_ref.astype(np.float32))
        ka = dw.k.cpu().view(torch.int16).numpy()
        for b, par in enumerate(w.trees):
            sl = w.nodes_of(b)
            path, nacc, bonus = oracle.verify_greedy(par, tokens[sl], greedy[sl])
            assert int(dw.accept_len[b]) == nacc and int(dw.bonus[b]) == bonus
            acc = dw.accepted[b].cpu().tolist()
            assert acc[:nacc] == path and all(x == -1 for x in acc[nacc:])
            for l in range(cfg.layers):
                ref, new_ctx = oracle.kv_compact(w.seq_view(k_before[l], b), path, int(w.ctx_lens[b]))
                assert int(dw.new_ctx[b]) == new_ctx
                assert np.array_equal(w.seq_view(ka[l], b)[:new_ctx], ref[:new_ctx])
        first = _step_outputs(dw)
        # a second step on the same buffers (the counters are cleared per step): the same top-k
        # and verdicts
        prev = ptd.step_topk_policy(ptd.STEP_TOPK_CLUSTERED if kind == "clustered" else ptd.STEP_TOPK_STREAMED)
        try:
            assert dw.step() == launches
            torch.cuda.synchronize()
        finally:
            ptd.step_topk_policy(prev)
        second = _step_outputs(dw)
        for key in ("idx", "val", "acc", "alen", "bonus", "status"):
            assert (first[key] == second[key]) if isinstance(first[key], int) else torch.equal(first[key], second[key])
        outs.append(second)
    a = outs[0]
    for b in outs[1:]:
        for key in a:
            if isinstance(a[key], int):
                assert a[key] == b[key], key
            else:
                assert torch.equal(a[key], b[key]), key
