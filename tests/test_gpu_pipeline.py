"""ptd_pipeline_*: host-buffer steps with copies overlapped with compute must give, step for
step, exactly what the synchronous ptd_tree_verify_step_host gives (same inputs, same order,
each on its own copy of the cache, which compaction changes every step)."""
import numpy as np
import pytest
import torch

from paper_2607_10661_gb300 import ptd
from paper_2607_10661_gb300 import synthetic as syn
from paper_2607_10661_gb300.harness import DeviceWorkload

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    import __graft_entry__

    __graft_entry__.build()


def _io(w, dw, step):
    """Pinned host inputs of one step (inputs vary with the step) and fresh output buffers."""
    c = w.cfg
    g = torch.Generator()
    g.manual_seed(100 + step)
    N, L = w.n_total, c.layers
    pin = lambda t: t.contiguous().pin_memory()
    t = dict(q_h=pin(torch.randn((L, N, c.hq, c.d), generator=g).to(torch.bfloat16)),
             logits_h=pin((torch.randn((N, c.vocab), generator=g) * 2).to(torch.bfloat16)),
             tokens_h=pin(torch.randint(0, c.vocab, (N,), generator=g, dtype=torch.int32)),
             parents_h=pin(dw.parents.cpu()), node_offsets_h=pin(dw.node_offsets.cpu()),
             ctx_lens_h=pin(dw.ctx_lens.cpu()),
             tree_k_h=pin(torch.randn((L, N, c.hkv, c.d), generator=g).to(torch.bfloat16)),
             tree_v_h=pin(torch.randn((L, N, c.hkv, c.d), generator=g).to(torch.bfloat16)),
             topk_idx_h=pin(torch.full((N, c.k), -1, dtype=torch.int32)),
             topk_val_h=pin(torch.zeros((N, c.k), dtype=torch.float32)),
             accepted_h=pin(torch.full((c.batch, w.max_nodes), -9, dtype=torch.int32)),
             accept_len_h=pin(torch.full((c.batch,), -9, dtype=torch.int32)),
             bonus_h=pin(torch.full((c.batch,), -9, dtype=torch.int32)),
             new_ctx_h=pin(torch.full((c.batch,), -9, dtype=torch.int32)),
             status_h=pin(torch.full((1,), -9, dtype=torch.int32)))
    # let some drafts match the argmax of their parent row, so that paths get accepted
    lg = t["logits_h"].float()
    par = t["parents_h"]
    for i in range(1, N):
        if i % 2:
            t["tokens_h"][i] = int(lg[int(par[i])].argmax())
    return t


OUT = ("topk_idx_h", "topk_val_h", "accepted_h", "accept_len_h", "bonus_h", "new_ctx_h", "status_h")


def test_pipeline_equals_synchronous_steps():
    w = syn.Workload(syn.shrink(syn.CONFIGS["llama3-8b-gqa"], layers=4, ctx=(300, 300), vocab=5000), 91)
    dw_a, dw_ref = DeviceWorkload(w), DeviceWorkload(w)
    tree_b, bufs_b = dw_a.twin_step_buffers()
    c = w.cfg
    steps = 6
    ios_p = [_io(w, dw_ref, s) for s in range(steps)]
    ios_r = [{k: (v.clone().pin_memory() if k in OUT else v) for k, v in t.items()} for t in ios_p]
    # reference: the synchronous host-buffer step, one at a time
    for s in range(steps):
        ptd.tree_verify_step_host(dw_ref.tree, dw_ref.cache, dw_ref.bufs, ptd.HostIO(**ios_r[s]))
        torch.cuda.synchronize()
    # pipelined: all steps submitted, two in flight
    n = 2 * c.layers * w.n_total * c.hkv * c.d * 2
    staging = [torch.empty(n, dtype=torch.uint8, device="cuda") for _ in range(2)]
    pipe = ptd.Pipeline(dw_a.cache, (dw_a.tree, tree_b), (dw_a.bufs, bufs_b), staging)
    hios = [ptd.HostIO(**t) for t in ios_p]
    tickets = []
    for s in range(steps):
        tickets.append(pipe.submit(hios[s]))
        if s >= 1:
            pipe.wait(tickets[s - 1])
    pipe.wait(tickets[-1])
    pipe.close()
    for s in range(steps):
        for k in OUT:
            assert torch.equal(ios_p[s][k], ios_r[s][k]), (s, k)
        assert int(ios_p[s]["status_h"][0]) == 0
    assert max(int(t["accept_len_h"][0]) for t in ios_r) >= 2
    torch.cuda.synchronize()
    assert torch.equal(dw_a.k, dw_ref.k) and torch.equal(dw_a.v, dw_ref.v)


def test_pipeline_argument_checks():
    w = syn.Workload(syn.shrink(syn.CONFIGS["llama3-8b-gqa"], layers=2, ctx=(64, 64), vocab=100), 92)
    dw_a = DeviceWorkload(w)
    tree_b, bufs_b = dw_a.twin_step_buffers()
    small = [torch.empty(16, dtype=torch.uint8, device="cuda") for _ in range(2)]
    with pytest.raises(ptd.PtdError) as e:
        ptd.Pipeline(dw_a.cache, (dw_a.tree, tree_b), (dw_a.bufs, bufs_b), small)
    assert e.value.status == ptd.WORKSPACE


def test_pipeline_submit_rejects_a_bad_host_tree_layout():
    """A host offset array that does not describe the slot's tree is refused with nothing
    enqueued and no ticket used: the next good submission gets ticket 0 and the right result."""
    w = syn.Workload(syn.shrink(syn.CONFIGS["llama3-8b-gqa"], layers=2, ctx=(200, 200), vocab=3000), 93)
    dw_a, dw_ref = DeviceWorkload(w), DeviceWorkload(w)
    tree_b, bufs_b = dw_a.twin_step_buffers()
    c = w.cfg
    n = 2 * c.layers * w.n_total * c.hkv * c.d * 2
    staging = [torch.empty(n, dtype=torch.uint8, device="cuda") for _ in range(2)]
    pipe = ptd.Pipeline(dw_a.cache, (dw_a.tree, tree_b), (dw_a.bufs, bufs_b), staging)
    good = _io(w, dw_ref, 0)
    for bad_offs in ([1, w.n_total], [0, w.n_total + 5], [0, w.n_total - 1]):
        bad = dict(good)
        bad["node_offsets_h"] = torch.tensor(bad_offs, dtype=torch.int32).pin_memory()
        with pytest.raises(ptd.PtdError) as e:
            pipe.submit(ptd.HostIO(**bad))
        assert e.value.status == ptd.INVALID_ARG
    ref = {k: (v.clone().pin_memory() if k in OUT else v) for k, v in good.items()}
    ptd.tree_verify_step_host(dw_ref.tree, dw_ref.cache, dw_ref.bufs, ptd.HostIO(**ref))
    torch.cuda.synchronize()
    assert pipe.submit(ptd.HostIO(**good)) == 0
    pipe.wait(0)
    pipe.close()
    for k in OUT:
        assert torch.equal(good[k], ref[k]), k
