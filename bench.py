"""Benchmark of the PTD tree-verify step on GB300.

One step = the whole hot path on one batch of synthetic input: tree-masked attention over
all 32 layers of the KV cache, per-node top-k of the logits, greedy verification and KV
compaction, through the C ABI (libptd.so), on the Llama-3-8B-shaped GQA workload
(32 query / 8 KV heads, head dim 128, committed context 8192, 63-node draft tree,
vocabulary 128256, top-4).

    python bench.py [--gpus N] [--steps K] [--warmup W] [--impl reference]

Prints one JSON line (rank 0).  `value` is whole-job steps/s with inputs resident in HBM,
the entry points called one by one with CUDA events around every attention launch (the
`roofline` figures come from those events); `step_call` is the same step through the
one-call entry ptd_tree_verify_step; `e2e` is the same metric through the pipelined
host-buffer API (ptd_pipeline_*: every step's inputs uploaded from pinned host memory and its
results read back by the host), with the one-step host call (a stream sync per step) beside
it.  Every step reads ~1.13 GB (more than the 129 MB L2), so no step finds the previous
one's data in L2.  Under torchrun each rank runs an independent replica (the step has no
cross-sequence exchange), timing is max over ranks, and value sums all ranks' steps.
`cpu_baseline` and `--impl reference` time the CPU oracle on a bounded sample of the same
workload, one process per host core.
"""
from __future__ import annotations

import argparse
import json
import os
import subprocess
import sys
import threading
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

WORKLOAD = "llama3-8b-gqa"
# dram__bytes_read.sum + dram__bytes_write.sum per launch from one ncu capture of the full
# Llama-3-8B-shaped workload (the attention: median of 20 launches of the one-pass launch
# list), keyed by the kernel source's sha256 prefix: a changed kernel reports null until it
# is captured again
PROFILED_ATTENTION_TRAFFIC = {"367a999933f00987": 1161794560}
PROFILED_LM_HEAD_TRAFFIC = {"541fa109411fd935": 1053963264}
MEASURED_PEAKS = os.path.join(ROOT, "MEASURED_PEAKS.json")
FALLBACK_HBM_GBS = 6800.0
NOMINAL_HBM_GBS = 8000.0


def _workload_desc(cfg) -> str:
    return (f"{cfg.name}: {cfg.layers} layers, {cfg.hq}q/{cfg.hkv}kv heads, head_dim {cfg.d}, "
            f"context {cfg.ctx[0]}, draft tree {cfg.nodes[0]} nodes (branching {','.join(map(str, cfg.branching))} "
            f"pruned), vocab {cfg.vocab}, top-{cfg.k}, batch {cfg.batch}")


def step_bytes(w) -> dict:
    """Algorithmic bytes of one step: every byte the step must move at least once."""
    c = w.cfg
    es = 2 if c.dtype == "bf16" else 4
    kv = sum(int(s) for s in w.seq_lens) * c.hkv * c.d * es * 2 * c.layers   # K and V, context + tree
    qo = 2 * c.layers * w.n_total * c.hq * c.d * es                          # Q read, O written
    logits = w.n_total * c.vocab * es
    return dict(kv=kv, qo=qo, logits=logits, attention=kv + qo, roofline=kv + logits)


def attention_flops(w) -> float:
    """QK^T and PV over every visible key (context plus the node's ancestors)."""
    c = w.cfg
    total = 0
    for b, par in enumerate(w.trees):
        depth = np.zeros(len(par), np.int64)
        for i in range(1, len(par)):
            depth[i] = depth[par[i]] + 1
        keys = len(par) * int(w.ctx_lens[b]) + int((depth + 1).sum())
        total += keys
    return 4.0 * c.d * c.hq * c.layers * total


# ----------------------------------------------------------------------------- clocks
class ClockSampler:
    QUERY = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
             "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
             "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, index: int):
        self.index = index
        self.proc = None
        self.lines = []

    def start(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.index), f"--query-gpu={self.QUERY}", "--format=csv,noheader,nounits",
                 "-lms", "100"], stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            self.thread = threading.Thread(target=self._read, daemon=True)
            self.thread.start()
        except OSError:
            self.proc = None

    def _read(self):
        for line in self.proc.stdout:
            self.lines.append((time.time(), line.strip()))

    def stop(self):
        if self.proc is not None:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()

    def summary(self, t0: float, t1: float) -> dict:
        rows = []
        for ts, line in self.lines:
            parts = [x.strip() for x in line.split(",")]
            if len(parts) < 8:
                continue
            try:
                rows.append((ts, float(parts[0]), float(parts[1]), parts[3:]))
            except ValueError:
                continue
        inside = [r for r in rows if t0 <= r[0] <= t1] or rows
        if not inside:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["no samples"]}
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = set()
        for r in inside:
            for n, v in zip(names, r[3][1:5]):
                if v.lower() == "active":
                    reasons.add(n)
        return {"sm_mhz": float(np.median([r[1] for r in inside])), "sm_max_mhz": max(r[2] for r in inside),
                "reasons": sorted(reasons), "samples": len(inside)}


def _profiled_traffic(table: dict, source: str):
    import hashlib

    with open(os.path.join(ROOT, "paper_2607_10661_gb300", "csrc", source), "rb") as f:
        return table.get(hashlib.sha256(f.read()).hexdigest()[:16])


def _attention_traffic(layers: int):
    t = _profiled_traffic(PROFILED_ATTENTION_TRAFFIC, "attention_tc.cu")
    return None if t is None or layers != 32 else t


def reduce_over_ranks(dist, values, device="cpu"):
    """Each value's maximum over the ranks (every rank gets it); the values themselves with
    one process.  The timed steps of every rank are bracketed by barriers, so the slowest
    rank's time is the job's."""
    if dist is None:
        return [float(v) for v in values]
    import torch

    t = torch.tensor([float(v) for v in values], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return [float(x) for x in t]


def aggregate_rate(world: int, steps: int, ms: float) -> float:
    """Whole-job steps/s: every rank ran `steps` steps of its own replica in `ms` (max)."""
    return world * steps / (ms * 1e-3)


def _peak_hbm():
    try:
        with open(MEASURED_PEAKS) as f:
            return float(json.load(f)["hbm_gbs"]), "measured"
    except Exception:
        return FALLBACK_HBM_GBS, "fallback"


# ----------------------------------------------------------------------------- GPU arm
def run_gpu(args, rank: int, world: int, dist):
    import torch

    from paper_2607_10661_gb300 import ptd
    from paper_2607_10661_gb300 import synthetic as syn
    from paper_2607_10661_gb300.harness import DeviceWorkload

    local = int(os.environ.get("LOCAL_RANK", "0"))
    torch.cuda.set_device(local)
    import __graft_entry__

    if rank == 0 or not os.path.exists(ptd.LIB_PATH):
        __graft_entry__.build()
    if dist is not None:
        dist.barrier()
    cfg = syn.CONFIGS[WORKLOAD]
    if args.layers:
        cfg = syn.shrink(cfg, layers=args.layers)
    w = syn.Workload(cfg, 1000 + rank)
    dw = DeviceWorkload(w, device=f"cuda:{local}")
    stream = torch.cuda.current_stream()
    nb = step_bytes(w)
    sampling = args.verify == "sampling"
    if sampling:
        # Alg. 2 at temperature 1: the uniforms are inputs of the step, like the logits
        gu = torch.Generator(device=f"cuda:{local}")
        gu.manual_seed(5000 + rank)
        u_acc = torch.rand(w.n_total, device=f"cuda:{local}", generator=gu)
        u_bon = torch.rand(cfg.batch, device=f"cuda:{local}", generator=gu)
    if args.lm_head:
        # the LM head feeds top-k from the nodes' hidden states: W [vocab][d_model] bf16 and H
        # [N_tot][d_model] (synthetic, seeded; Llama-3-8B's head is 128256 x 4096)
        d_model = 4096
        gh = torch.Generator(device=f"cuda:{local}")
        gh.manual_seed(7000 + rank)
        lm_w = (torch.randn((cfg.vocab, d_model), generator=gh, device=f"cuda:{local}") / d_model ** 0.5).to(
            torch.bfloat16)
        lm_h = torch.randn((w.n_total, d_model), generator=gh, device=f"cuda:{local}").to(torch.bfloat16)
        lm_ws = torch.empty(ptd.lm_head_workspace_size(w.n_total, cfg.vocab), dtype=torch.uint8,
                            device=f"cuda:{local}")
        lm_evs = []
    if args.ptd_step:
        args.draft_update = True
        # the tree's own (unrotated) K and V of every layer, written by the rotary step into
        # the cache slots the attention reads; the candidate pool the draft tree feeds
        gk = torch.Generator(device=f"cuda:{local}")
        gk.manual_seed(6000 + rank)
        tree_k = torch.randn((cfg.layers, w.n_total, cfg.hkv, cfg.d), generator=gk,
                             device=f"cuda:{local}").to(dw.tdtype)
        tree_v = torch.randn_like(tree_k)
        pool = ptd.CandidatePool(1 << 20, device=f"cuda:{local}")
        ret = [torch.zeros(1, dtype=torch.int32, device=f"cuda:{local}"),
               torch.empty(ptd.MAX_TREE_NODES, dtype=torch.int32, device=f"cuda:{local}"),
               torch.empty(ptd.MAX_TREE_NODES, dtype=torch.int32, device=f"cuda:{local}")]
        pool_step = [0]
    if args.draft_update:
        # the step's tree as a one-seed draft forest, grown by every node's top-1 (width 4,
        # depth 6: the paper's best setting); the output is the next step's draft tree
        if cfg.batch != 1:
            raise SystemExit("--draft-update times the one-tree workload only")
        du_dev = f"cuda:{local}"
        du_cnt = torch.tensor([w.n_total], dtype=torch.int32, device=du_dev)
        du_out = [torch.empty((1,), dtype=torch.int32, device=du_dev)] + \
                 [torch.empty((1, ptd.MAX_TREE_NODES), dtype=torch.int32, device=du_dev) for _ in range(3)] + \
                 [torch.empty((1, w.n_total), dtype=torch.int32, device=du_dev)]

    def one_step(ev=None):
        n = 0
        if args.ptd_step:   # positions C + |pi(v)| - 1, rotary encoding, tree K/V into the cache
            n += ptd.tree_rope_append(dw.tree, dw.cache, 0, dw.q, cfg.hq, tree_k, tree_v, 500000.0, dw.dev_status)
        if ev is not None:
            ev[0].record(stream)
        n += dw.attention()
        if ev is not None:
            ev[1].record(stream)
        if args.lm_head:
            if ev is not None:
                e2 = (torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
                e2[0].record(stream)
            n += ptd.lm_head_topk(lm_h, lm_w, cfg.k, dw.topk_idx, dw.topk_val, lm_ws, dw.dev_status)
            if ev is not None:
                e2[1].record(stream)
                lm_evs.append(e2)
        else:
            n += dw.topk()
        if args.draft_update:
            n += ptd.draft_tree_update(du_cnt, dw.parents.view(1, -1), dw.tokens.view(1, -1), dw.topk_idx, 1, 4, 6,
                                       ptd.MAX_TREE_NODES, *du_out, dw.dev_status)
        if args.ptd_step:   # the grown draft tree joins the pool; C_X for the next step
            pool_step[0] += 1
            n += pool.merge(pool_step[0], du_out[0], du_out[1][0], du_out[2][0], dw.dev_status, max_load=1 << 19)
        if sampling:
            n += ptd.verify_sampling(dw.tree, dw.tokens, dw.logits, 1.0, u_acc, u_bon, dw.accepted, dw.accept_len,
                                     dw.bonus, dw.dev_status)
            n += dw.compact()
        else:
            n += dw.verify_and_compact()
        if args.ptd_step:
            n += pool.retrieve(dw.bonus[:1], 4, 6, 64, *ret)
        return n

    dw.dev_status.zero_()              # sticky status word: cleared once, read after the run
    sampler = ClockSampler(local)
    sampler.start()
    time.sleep(0.5)
    for _ in range(args.warmup):
        one_step()
    torch.cuda.synchronize()
    assert int(dw.dev_status.item()) == 0, ptd.status_string(int(dw.dev_status.item()))

    K = args.steps
    evs = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(K)]
    start, end = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    if dist is not None:
        dist.barrier()
    torch.cuda.synchronize()
    t_wall0 = time.time()
    start.record(stream)
    launches = 0
    for i in range(K):
        launches += one_step(evs[i])
    end.record(stream)
    torch.cuda.synchronize()
    t_wall1 = time.time()
    if dist is not None:
        dist.barrier()
    ms = start.elapsed_time(end)
    attn_ms = float(np.mean([a.elapsed_time(b) for a, b in evs]))
    lm_ms = float(np.mean([a.elapsed_time(b) for a, b in lm_evs])) if args.lm_head else None
    clocks = sampler.summary(t_wall0, t_wall1)
    sampler.stop()
    status = int(dw.dev_status.item())

    # ---- the same step through its one-call entry (ptd_tree_verify_step), with no events
    # between its launches: there the top-k may start while the attention grid drains
    step_call_ms, Kc = None, max(10, K // 4)
    if not (args.lm_head or args.draft_update or args.ptd_step or sampling):
        for _ in range(3):
            ptd.tree_verify_step(dw.tree, dw.cache, dw.bufs, stream)
        c0, c1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        if dist is not None:
            dist.barrier()
        torch.cuda.synchronize()
        c0.record(stream)
        for _ in range(Kc):
            ptd.tree_verify_step(dw.tree, dw.cache, dw.bufs, stream)
        c1.record(stream)
        torch.cuda.synchronize()
        step_call_ms = c0.elapsed_time(c1)
        status |= int(dw.dev_status.item())

    # ---- end to end: pinned host inputs and outputs through ptd_tree_verify_step_host
    N, L = w.n_total, cfg.layers
    C = int(w.ctx_lens[0])
    pin = lambda t: t.contiguous().pin_memory()
    io_t = dict(q_h=pin(dw.q.cpu()), logits_h=pin(dw.logits.cpu()), tokens_h=pin(dw.tokens.cpu()),
                parents_h=pin(dw.parents.cpu()), node_offsets_h=pin(dw.node_offsets.cpu()),
                ctx_lens_h=pin(dw.ctx_lens.cpu()),
                tree_k_h=pin(dw.k[:, 0, C:C + N].cpu()), tree_v_h=pin(dw.v[:, 0, C:C + N].cpu()),
                topk_idx_h=pin(torch.zeros((N, cfg.k), dtype=torch.int32)),
                topk_val_h=pin(torch.zeros((N, cfg.k), dtype=torch.float32)),
                accepted_h=pin(torch.zeros((cfg.batch, w.max_nodes), dtype=torch.int32)),
                accept_len_h=pin(torch.zeros(cfg.batch, dtype=torch.int32)),
                bonus_h=pin(torch.zeros(cfg.batch, dtype=torch.int32)),
                new_ctx_h=pin(torch.zeros(cfg.batch, dtype=torch.int32)),
                status_h=pin(torch.zeros(1, dtype=torch.int32)))
    io = ptd.HostIO(**io_t)
    h2d = sum(io_t[n].numel() * io_t[n].element_size() for n in
              ("q_h", "logits_h", "tokens_h", "parents_h", "node_offsets_h", "ctx_lens_h", "tree_k_h", "tree_v_h"))
    d2h = sum(io_t[n].numel() * io_t[n].element_size() for n in
              ("topk_idx_h", "topk_val_h", "accepted_h", "accept_len_h", "bonus_h", "new_ctx_h", "status_h"))
    for _ in range(3):
        ptd.tree_verify_step_host(dw.tree, dw.cache, dw.bufs, io)
        stream.synchronize()
    Ke = max(10, K // 5)
    if dist is not None:
        dist.barrier()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for _ in range(Ke):
        ptd.tree_verify_step_host(dw.tree, dw.cache, dw.bufs, io)
        stream.synchronize()             # the host reads the step's result before the next step
    e1.record(stream)
    torch.cuda.synchronize()
    sync_ms = e0.elapsed_time(e1)
    sync_ok = int(io_t["status_h"][0]) == 0
    # the same steps through the pipelined host-buffer API: step i + 1's uploads and step
    # i - 1's downloads overlap step i's computation; the host reads every step's result
    tree_b, bufs_b = dw.twin_step_buffers()
    stage_n = 2 * L * N * cfg.hkv * cfg.d * dw.k.element_size()
    staging = [torch.empty(stage_n, dtype=torch.uint8, device=f"cuda:{local}") for _ in range(2)]
    pipe = ptd.Pipeline(dw.cache, (dw.tree, tree_b), (dw.bufs, bufs_b), staging)
    io_t2 = {k: (pin(v.clone()) if k in ("topk_idx_h", "topk_val_h", "accepted_h", "accept_len_h", "bonus_h",
                                         "new_ctx_h", "status_h") else v) for k, v in io_t.items()}
    ios = [io, ptd.HostIO(**io_t2)]
    outs_t = [io_t, io_t2]

    def run_pipeline(n):
        ok, prev = True, None
        for i in range(n):
            tk = pipe.submit(ios[i & 1])
            if prev is not None:
                pipe.wait(prev)
                ok = ok and int(outs_t[(i - 1) & 1]["status_h"][0]) == 0
            prev = tk
        pipe.wait(prev)
        return ok and int(outs_t[(n - 1) & 1]["status_h"][0]) == 0

    run_pipeline(4)
    torch.cuda.synchronize()
    if dist is not None:
        dist.barrier()
    e0.record(stream)
    e2e_ok = run_pipeline(Ke) and sync_ok
    e1.record(stream)
    torch.cuda.synchronize()
    e2e_ms = e0.elapsed_time(e1)
    pipe.close()

    ms, e2e_ms, sync_ms, sc_ms = reduce_over_ranks(dist, [ms, e2e_ms, sync_ms, step_call_ms or 0.0],
                                                   f"cuda:{local}")
    step_call_ms = sc_ms if step_call_ms is not None else None

    peak, peak_kind = _peak_hbm()
    achieved = nb["attention"] / (attn_ms * 1e-3) / 1e9
    ms_step = ms / K
    value = aggregate_rate(world, K, ms)
    flops = attention_flops(w)
    out = {
        "metric": "tree-verify steps/sec (HBM GB/s and fraction of ~8 TB/s alongside)",
        "value": round(value, 3),
        "unit": "steps/s",
        "n_gpus": world,
        "steps": K,
        "warmup": args.warmup,
        "ms_per_step": round(ms_step, 5),
        "higher_is_better": True,
        "scaling": "weak",
        "vs_baseline": None,
        "dtype": "bf16",
        "data": "synthetic (seeded N(0,1) Q/K/V, N(0,2) logits with a planted +6 token, random pruned tree)",
        "config": {"workload": _workload_desc(cfg), "batch": cfg.batch, "layers": cfg.layers,
                   "context": cfg.ctx[0], "tree_nodes": w.n_total, "vocab": cfg.vocab, "k": cfg.k,
                   "verify": "sampling (Alg. 2, temperature 1)" if sampling else "greedy",
                   "draft_update": "top-1 expansion, width 4, depth 6 (Alg. 1 step 3)" if args.draft_update else None,
                   "top_k_source": ("LM head from hidden states (63 x 4096 by 128256 x 4096 bf16, logits not "
                                    "written)" if args.lm_head else "resident logits"),
                   "ptd_step": ("tree positions + rotary encoding + K/V append (32 layers), attention, top-k, "
                                "verification + compaction, draft update, pool merge, pool retrieval")
                   if args.ptd_step else None,
                   "parallelism": f"replicas x{world}" if world > 1 else "single GPU",
                   "l2": "inputs larger than L2 (%.2f GB read per step vs 129 MB L2)" % (nb["roofline"] / 1e9)},
        "step_roofline_bytes": nb["roofline"],
        "hbm_gbs": round(nb["roofline"] / (ms_step * 1e-3) / 1e9, 1),
        "hbm_frac_of_8tbs": round(nb["roofline"] / (ms_step * 1e-3) / 1e9 / NOMINAL_HBM_GBS, 4),
        "hbm_frac_of_measured": round(nb["roofline"] / (ms_step * 1e-3) / 1e9 / peak, 4),
        "roofline": {"bound": "hbm", "kernel": "tree_attn_tc_kernel", "achieved": round(achieved, 1),
                     "peak": peak, "peak_kind": peak_kind, "unit": "GB/s", "frac": round(achieved / peak, 4),
                     "traffic": _attention_traffic(cfg.layers), "bytes_per_launch": nb["attention"],
                     "avg_launch_ms": round(attn_ms, 5),
                     "tensor_tflops": round(flops / (attn_ms * 1e-3) / 1e12, 1)},
        "clocks": clocks,
        "step_call": (None if step_call_ms is None else
                      {"value": round(aggregate_rate(world, Kc, step_call_ms), 3), "unit": "steps/s", "steps": Kc,
                       "api": "ptd_tree_verify_step (device buffers, no events between the launches)"}),
        "e2e": {"value": round(aggregate_rate(world, Ke, e2e_ms), 3), "unit": "steps/s", "steps": Ke,
                "h2d_bytes_per_step": int(h2d), "d2h_bytes_per_step": int(d2h), "status_ok": e2e_ok,
                "verify": "greedy",
                "api": "ptd_pipeline_submit / ptd_pipeline_wait (uploads and downloads overlapped with compute, "
                       "two steps in flight); every step's inputs uploaded from pinned host memory and its result "
                       "read by the host",
                "one_step_call_value": round(aggregate_rate(world, Ke, sync_ms), 3)},
        "lm_head": ({"kernel": "lm_head_topk_kernel", "avg_launch_ms": round(lm_ms, 5),
                     "bytes_per_launch": int(lm_w.numel() * 2 + lm_h.numel() * 2),
                     "achieved_gbs": round((lm_w.numel() * 2 + lm_h.numel() * 2) / (lm_ms * 1e-3) / 1e9, 1),
                     "frac": round((lm_w.numel() * 2 + lm_h.numel() * 2) / (lm_ms * 1e-3) / 1e9
                                   / _peak_hbm()[0], 4), "peak_kind": _peak_hbm()[1],
                     "traffic": (_profiled_traffic(PROFILED_LM_HEAD_TRAFFIC, "lm_head.cu")
                                 if cfg.vocab == 128256 else None),
                     "note": "two launches: the product with per-CTA top-k, then the per-row merge"}
                    if args.lm_head else None),
        "gpu_launches": int(launches),
        "status": ptd.status_string(status),
    }
    if rank == 0 and not args.no_cpu_baseline:
        out["cpu_baseline"] = cpu_baseline(args.cpu_seconds, sampling)
    return out


# ----------------------------------------------------------------------------- CPU oracle
_SAMPLE_CODE = r"""
import json, sys, time
sys.path.insert(0, {root!r})
import numpy as np
import oracle
from paper_2607_10661_gb300 import synthetic as syn
cfg = syn.CONFIGS[{workload!r}]
w = syn.Workload(cfg, 1000)
G, C, L, H = cfg.hq // cfg.hkv, int(w.ctx_lens[0]), cfg.layers, cfg.hkv
lg = syn.widen(w.logits, "bf16")
cache = {{}}
def layer(l):
    if l not in cache:
        cache.clear()
        kl, vl = w.kv_layer(l)
        cache[l] = (syn.widen(w.q_layer(l), "bf16"), w.seq_view(syn.widen(kl, "bf16"), 0),
                    w.seq_view(syn.widen(vl, "bf16"), 0))
    return cache[l]
per_step = []
deadline = time.time() + {budget}
for i in range({warmup} + {steps}):
    j = i * {workers} + {worker}          # this process's share of the samples
    u = j % (L * H)
    q, k, v = layer(u // H)
    h = u % H
    t0 = time.time()
    oracle.tree_attention(q[:, h * G:(h + 1) * G], k[:, h:h + 1], v[:, h:h + 1], w.trees[0], C)
    t1 = time.time()
    idx, _ = oracle.topk(lg[j % w.n_total], cfg.k)
    t2 = time.time()
    if {sampling}:
        g = np.random.default_rng(j)
        path, n, bonus, _ = oracle.verify_sampling(w.trees[0], w.tokens, lg, 1.0, g.random(w.n_total), g.random())
    else:
        target = np.full(w.n_total, int(idx[0]), np.int64)
        path, n, bonus = oracle.verify_greedy(w.trees[0], w.tokens, target)
    t3 = time.time()
    oracle.kv_compact(k if j % 2 == 0 else v, path, C)
    t4 = time.time()
    if i >= {warmup}:
        per_step.append((t1 - t0) * L * H + (t2 - t1) * w.n_total + (t3 - t2) + (t4 - t3) * 2 * L)
    if time.time() > deadline and len(per_step) > 0:
        break
print(json.dumps(dict(per_step=per_step)))
"""

SAMPLE_DESC = ("per sample: one of the 256 (layer, KV head) attention units, one of the 63 top-k rows, the "
               "whole verification and compaction of one of the 64 layer K/V tensors, timed in one process "
               "(BLAS pinned to one thread) and scaled by those counts to one full step; one such process per "
               "host core, each on its own share of the samples, all running at once")


def host_cores() -> int:
    try:
        return len(os.sched_getaffinity(0))
    except AttributeError:
        return os.cpu_count() or 1


def oracle_samples(steps: int, warmup: int, budget_s: float, sampling: bool = False, workers: int = 1):
    """Per-process lists of per-sample full-step times (seconds): `workers` processes (fresh
    interpreters, never forked from one that touched the GPU) run the oracle at once."""
    env = dict(os.environ, OMP_NUM_THREADS="1", OPENBLAS_NUM_THREADS="1", MKL_NUM_THREADS="1",
               CUDA_VISIBLE_DEVICES="")
    per_worker = max(1, -(-int(steps) // workers))
    procs = []
    for wk in range(workers):
        code = _SAMPLE_CODE.format(root=ROOT, workload=WORKLOAD, budget=float(budget_s), steps=per_worker,
                                   warmup=int(warmup), sampling=bool(sampling), worker=wk, workers=workers)
        procs.append(subprocess.Popen([sys.executable, "-c", code], stdout=subprocess.PIPE,
                                      stderr=subprocess.PIPE, text=True, env=env))
    out = []
    for pr in procs:
        so, se = pr.communicate(timeout=budget_s * 4 + 300)
        if pr.returncode != 0:
            raise RuntimeError(se[-500:])
        out.append(json.loads(so.strip().splitlines()[-1])["per_step"])
    return out


def oracle_rate(per_worker) -> float:
    """Whole-host steps/s: the processes ran at the same time, each at 1 / (its mean step time)."""
    return float(sum(1.0 / np.mean(p) for p in per_worker))


def cpu_baseline(budget_s: float, sampling: bool = False) -> dict:
    """The oracle as it stands on a bounded sample of the workload (about budget_s of wall
    time), on every host core, and on one core alone."""
    cores = host_cores()
    try:
        one = oracle_samples(10000, 1, budget_s / 2, sampling)[0]
        many = oracle_samples(10000, 1, budget_s / 2, sampling, workers=cores)
    except Exception as e:  # reported, never fatal for the GPU line
        return {"value": None, "unit": "steps/s", "cores": cores, "kind": "oracle", "error": str(e)[-300:]}
    n = sum(len(p) for p in many)
    return {"value": oracle_rate(many), "unit": "steps/s", "cores": cores, "kind": "oracle",
            "sample": f"{n} samples over {cores} processes; " + SAMPLE_DESC,
            "single_core": {"value": 1.0 / float(np.mean(one)), "unit": "steps/s", "cores": 1,
                            "samples": len(one), "seconds_per_step": float(np.mean(one))}}


def run_reference(args):
    """--impl reference: the CPU oracle on the host cores, one bounded sample per step; the
    run stops early (reporting the steps it timed) once about --ref-seconds of samples are taken."""
    from paper_2607_10661_gb300 import synthetic as syn

    cfg = syn.CONFIGS[WORKLOAD]
    cores = host_cores()
    try:
        per = oracle_samples(args.steps, min(args.warmup, 1), args.ref_seconds, args.verify == "sampling",
                             workers=cores)
    except Exception as e:
        return {"impl": "reference", "unavailable": "oracle sample failed: " + str(e)[-200:]}
    value = oracle_rate(per)
    sec = 1.0 / value
    n = sum(len(p) for p in per)
    return {
        "impl": "reference",
        "metric": "tree-verify steps/sec (HBM GB/s and fraction of ~8 TB/s alongside)",
        "value": value, "unit": "steps/s", "n_gpus": args.gpus, "steps": n, "warmup": min(args.warmup, 1),
        "ms_per_step": sec * 1e3, "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
        "dtype": "f64", "data": "synthetic", "config": {"workload": _workload_desc(cfg)},
        "cpu_baseline": {"value": value, "unit": "steps/s", "cores": cores, "kind": "oracle",
                         "sample": f"{n} samples over {cores} processes; " + SAMPLE_DESC},
        "e2e": {"value": value, "unit": "steps/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=2000)
    ap.add_argument("--warmup", type=int, default=20)
    ap.add_argument("--impl", default="ptd", choices=["ptd", "reference"])
    ap.add_argument("--layers", type=int, default=0, help="override the layer count (profiling captures)")
    ap.add_argument("--cpu-seconds", type=float, default=20.0)
    ap.add_argument("--ref-seconds", type=float, default=150.0,
                    help="--impl reference: stop sampling the oracle after about this many seconds")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--lm-head", action="store_true",
                    help="top-k from the LM head (ptd_lm_head_topk, logits never written) instead of from "
                         "resident logits")
    ap.add_argument("--ptd-step", action="store_true",
                    help="the whole PTD step: rotary encoding and tree K/V append, the verify step, the draft "
                         "tree update and the candidate pool's merge and retrieval (Alg. 1 steps 1-6)")
    ap.add_argument("--draft-update", action="store_true",
                    help="add the draft tree update (Sec. 3.1 expansion and depth control) to every step")
    ap.add_argument("--verify", default="greedy", choices=["greedy", "sampling"],
                    help="verification strategy of the step (Sec. 3.2): greedy, or sampling (Alg. 2)")
    args = ap.parse_args()
    args.warmup = max(3, args.warmup)

    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    if args.impl == "reference":
        if rank == 0:
            print(json.dumps(run_reference(args)), flush=True)
        return
    dist = None
    if world > 1:
        import torch.distributed as dist_mod

        dist_mod.init_process_group("nccl")
        dist = dist_mod
    out = run_gpu(args, rank, world, dist)
    if rank == 0:
        print(json.dumps(out), flush=True)
    if dist is not None:
        dist.destroy_process_group()


if __name__ == "__main__":
    main()
