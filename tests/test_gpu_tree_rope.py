"""ptd_tree_rope_append on the GPU against the oracle (Sec. 3.1 "Tree Construction": a
node's position is set by |pi(v)|): positions bit-exact; rotated queries and keys within
the step's tolerance of the float64 rotation (bf16: max-abs 2e-2, mean-abs 2e-3; fp32:
1e-4); values copied bit for bit; every other cache row untouched."""
import numpy as np
import pytest
import torch

import oracle
from paper_2607_10661_gb300 import ptd
from paper_2607_10661_gb300 import synthetic as syn
from paper_2607_10661_gb300.harness import DeviceWorkload

pytestmark = pytest.mark.gpu

CASES = {
    # name: (config, overrides, rope base, layer)
    "llama2-mha-contiguous": ("llama2-7b-layer", dict(ctx=(2048, 2048), vocab=100), 10000.0, 0),
    "llama3-gqa-layer5": ("llama3-8b-gqa", dict(layers=6, ctx=(8192, 8192), vocab=100), 500000.0, 5),
    "batched-paged": ("batched-paged", dict(vocab=100, layers=2), 500000.0, 1),
    "tiny-fp32": ("tiny-fp32", {}, 10000.0, 0),
    "long-context": ("long-context", dict(vocab=100), 1000000.0, 0),
}


@pytest.fixture(scope="module", autouse=True)
def _built():
    import __graft_entry__

    __graft_entry__.build()


def _run(name, ctx_override=None):
    base_cfg, over, base, layer = CASES[name]
    w = syn.Workload(syn.shrink(syn.CONFIGS[base_cfg], **over), 61)
    dw = DeviceWorkload(w, with_step_buffers=False)
    c = w.cfg
    if ctx_override is not None:
        dw.ctx_lens.copy_(torch.tensor(ctx_override, dtype=torch.int32))
    g = torch.Generator(device="cuda")
    g.manual_seed(62)
    q = torch.randn((w.n_total, c.hq, c.d), generator=g, device="cuda").to(dw.tdtype)
    k = torch.randn((w.n_total, c.hkv, c.d), generator=g, device="cuda").to(dw.tdtype)
    v = torch.randn((w.n_total, c.hkv, c.d), generator=g, device="cuda").to(dw.tdtype)
    q0, k_before, v_before = q.clone(), dw.k.clone(), dw.v.clone()
    pos = torch.full((w.n_total,), -1, dtype=torch.int32, device="cuda")
    assert ptd.tree_rope_append(dw.tree, dw.cache, layer, q, c.hq, k, v, base, dw.dev_status, pos) == 1
    torch.cuda.synchronize()
    return w, dw, layer, base, q0, q, k, v, k_before, v_before, pos


def _close(got, want, dtype):
    err = np.abs(got - want)
    if dtype == "bf16":
        assert err.max() <= 2e-2 and err.mean() <= 2e-3, (err.max(), err.mean())
    else:
        assert err.max() <= 1e-4, err.max()


@pytest.mark.parametrize("name", list(CASES))
def test_tree_rope_append_matches_oracle(name):
    w, dw, layer, base, q0, q, k, v, k_before, v_before, pos = _run(name)
    c = w.cfg
    assert int(dw.dev_status.item()) == 0
    ctx = dw.ctx_lens.cpu().numpy()
    want_pos = np.concatenate([oracle.tree_positions(w.trees[b], int(ctx[b])) for b in range(c.batch)])
    assert pos.cpu().numpy().tolist() == want_pos.tolist()
    _close(q.float().cpu().numpy(), oracle.rope(q0.float().cpu().numpy(), want_pos, base), c.dtype)
    kc, vc = dw.k.cpu(), dw.v.cpu()
    kb, vb = k_before.cpu(), v_before.cpu()
    k_rot = oracle.rope(k.float().cpu().numpy(), want_pos, base)
    written = torch.zeros(kc.shape[:-2], dtype=torch.bool)
    for b in range(c.batch):
        sl = w.nodes_of(b)
        o, i = w.slot_rows(b, int(ctx[b]) + len(w.trees[b]))
        o, i = o[int(ctx[b]):], i[int(ctx[b]):]
        _close(kc[layer, o, i].float().numpy(), k_rot[sl], c.dtype)
        assert torch.equal(vc[layer, o, i], v[sl].cpu())
        written[layer, o, i] = True
    assert torch.equal(kc[~written], kb[~written]) and torch.equal(vc[~written], vb[~written])


def test_slots_outside_the_cache_are_refused_node_by_node():
    """A context that leaves no room for the last two nodes: those write nothing and the
    status says so; the nodes that fit are written as usual."""
    base_cfg, over, base, layer = CASES["llama2-mha-contiguous"]
    w = syn.Workload(syn.shrink(syn.CONFIGS[base_cfg], **over), 61)
    cap = w.seq_capacity
    T = len(w.trees[0])
    w2, dw, layer, base, q0, q, k, v, k_before, v_before, pos = _run("llama2-mha-contiguous", [cap - T + 2])
    assert int(dw.dev_status.item()) == ptd.INVALID_TREE
    kc, kb = dw.k.cpu(), k_before.cpu()
    C = cap - T + 2
    assert not torch.equal(kc[layer, 0, C:cap], kb[layer, 0, C:cap])       # the first T - 2 nodes landed
    assert torch.equal(kc[layer, 0, :C], kb[layer, 0, :C])


def test_layer_range_in_one_launch():
    """Every layer of the Llama-3-8B-shaped stack in one launch equals the layers one by one."""
    w = syn.Workload(syn.shrink(syn.CONFIGS["llama3-8b-gqa"], layers=4, ctx=(300, 300), vocab=100), 63)
    c = w.cfg
    dws = [DeviceWorkload(w, with_step_buffers=False) for _ in range(2)]
    g = torch.Generator(device="cuda")
    g.manual_seed(64)
    q = torch.randn((c.layers, w.n_total, c.hq, c.d), generator=g, device="cuda").to(torch.bfloat16)
    k = torch.randn((c.layers, w.n_total, c.hkv, c.d), generator=g, device="cuda").to(torch.bfloat16)
    v = torch.randn((c.layers, w.n_total, c.hkv, c.d), generator=g, device="cuda").to(torch.bfloat16)
    qa, qb = q.clone(), q.clone()
    assert ptd.tree_rope_append(dws[0].tree, dws[0].cache, 0, qa, c.hq, k, v, 500000.0, dws[0].dev_status) == 1
    for l in range(c.layers):
        ptd.tree_rope_append(dws[1].tree, dws[1].cache, l, qb[l], c.hq, k[l], v[l], 500000.0, dws[1].dev_status)
    torch.cuda.synchronize()
    assert torch.equal(qa, qb) and torch.equal(dws[0].k, dws[1].k) and torch.equal(dws[0].v, dws[1].v)
    assert int(dws[0].dev_status.item()) == 0 and int(dws[1].dev_status.item()) == 0
