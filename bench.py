"""Benchmark of the PTD tree-verify step on GB300.

One step = the whole hot path on one batch of synthetic input: tree-masked attention over
every layer of the KV cache, per-node top-k of the logits, greedy verification and KV
compaction, through the C ABI (libptd.so).  The workload is one of the five seeded synthetic
configurations (`--workload`); the default is the Llama-3-8B-shaped GQA stack (32 query / 8
KV heads, head dim 128, 32 layers, committed context 8192, 63-node draft tree, vocabulary
128256, top-4), the configuration the 70 % HBM target is stated for.

    python bench.py [--gpus N] [--steps K] [--warmup W] [--workload NAME] [--impl reference]

Prints one JSON line (rank 0).
  value      whole-job steps/s through the one-call entry ptd_tree_verify_step, inputs
             resident in HBM: K steps captured in a CUDA graph (so that the host's launch
             cost is not what is timed) and replayed between CUDA events, the region repeated
             until at least one second of wall time has passed, the median region reported.
             Workloads whose step reads less than three times the L2 size get that many copies
             of every buffer, used in turn, so that no step finds its inputs in L2.  `eager`
             is the same steps called from Python one by one.
  roofline   the attention kernel's algorithmic bytes (or FLOPs) over its mean launch time,
             from timing events (graph nodes) around every attention launch of a second,
             equally repeated loop that calls the step's entry points one by one.
  e2e        the same metric through the pipelined host-buffer API (ptd_pipeline_*): every
             step's inputs uploaded from pinned host memory and its results read back.
  clocks     SM clock and throttle reasons sampled every 10 ms through NVML, only inside
             the timed regions.
  cpu_baseline / --impl reference
             the CPU oracle, whole steps (every attention unit, every top-k row, the
             verification on this step's own greedy targets, the compaction of every layer),
             spread over the host cores by worker processes started with spawn.
Under torchrun each rank runs an independent replica (the step has no cross-sequence
exchange), timing is the maximum over ranks, and value sums all ranks' steps.
"""
from __future__ import annotations

import argparse
import ctypes
import json
import os
import statistics
import sys
import threading
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

DEFAULT_WORKLOAD = "llama3-8b-gqa"
METRIC = "tree-verify steps/sec (HBM GB/s and fraction of ~8 TB/s alongside)"
# dram__bytes_read.sum + dram__bytes_write.sum per attention launch from one ncu capture,
# keyed by (workload, the kernel source's sha256 prefix): a changed kernel reports null
# until it is captured again
PROFILED_ATTENTION_TRAFFIC = {(("llama3-8b-gqa", 32), "766310cc72ef5798"): 1112748032}
PROFILED_LM_HEAD_TRAFFIC = {"c177b463ccbf468a": 1056910592}
MEASURED_PEAKS = os.path.join(ROOT, "MEASURED_PEAKS.json")
# the tail of the one-call step (ptd_step_tail)
STEP_TAILS = {0: "top-k, then verification + compaction in one launch",
              1: "clustered top-k (one cluster per row) verifying the trees, then a compaction kernel",
              2: "streamed top-k (rows back to back, one share per CTA) verifying the trees, then a compaction kernel"}
FALLBACK_HBM_GBS = 6800.0
FALLBACK_BF16_TFLOPS_SUSTAINED = 1700.0
NOMINAL_HBM_GBS = 8000.0
MIN_REGION_WALL_S = 1.0


def workload_desc(cfg) -> str:
    ctx = f"{cfg.ctx[0]}" if cfg.ctx[0] == cfg.ctx[1] else f"{cfg.ctx[0]}-{cfg.ctx[1]} (uniform, per sequence)"
    nodes = f"{cfg.nodes[0]}" if cfg.nodes[0] == cfg.nodes[1] else f"{cfg.nodes[0]}-{cfg.nodes[1]}"
    shape = (f"branching {','.join(map(str, cfg.branching))} pruned" if cfg.tree == "branching" else
             "complete binary" if cfg.tree == "binary" else
             f"random depth {cfg.depth_range[0]}-{cfg.depth_range[1]}" if cfg.tree == "random-depth" else cfg.tree)
    cache = f", paged cache of {cfg.page_size}-token pages" if cfg.page_size else ""
    return (f"{cfg.name}: {cfg.layers} layers, {cfg.hq}q/{cfg.hkv}kv heads, head_dim {cfg.d}, context {ctx}, "
            f"draft tree {nodes} nodes ({shape}), vocab {cfg.vocab}, top-{cfg.k}, batch {cfg.batch}{cache}, "
            f"{cfg.dtype}")


def bench_config(w, extra: dict | None = None) -> dict:
    """The `config` object of both arms' lines (the same workload, the same dict)."""
    c = w.cfg
    out = {"workload": workload_desc(c), "batch": c.batch, "layers": c.layers,
           "context": [int(x) for x in w.ctx_lens], "tree_nodes": int(w.n_total), "vocab": c.vocab, "k": c.k,
           "seed": int(w.seed)}
    out.update(extra or {})
    return out


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
    """SM clock, power and throttle reasons of one GPU every `period_s`, through NVML (read
    only).  summary(regions) keeps only the samples taken inside the given wall-clock
    intervals and says "no samples" when none fell there."""

    _REASONS = {0x4: "sw_power_cap", 0x8: "hw_slowdown", 0x20: "sw_thermal_slowdown", 0x40: "hw_thermal_slowdown",
                0x80: "hw_power_brake_slowdown"}

    def __init__(self, torch_index: int, period_s: float = 0.01):
        self.period = period_s
        self.samples = []
        self.source = None
        self._stop = threading.Event()
        self._thread = None
        self._nvml = None
        self._h = None
        try:
            self._open(torch_index)
        except Exception as e:  # reported in the line, never fatal
            self.source = f"unavailable ({e})"[:120]

    def _open(self, torch_index):
        import torch

        nv = ctypes.CDLL("libnvidia-ml.so.1")
        if nv.nvmlInit_v2() != 0:
            raise RuntimeError("nvmlInit failed")
        h = ctypes.c_void_p()
        props = torch.cuda.get_device_properties(torch_index)
        found = False
        try:
            bus = b"%08X:%02X:%02X.0" % (props.pci_domain_id, props.pci_bus_id, props.pci_device_id)
            found = nv.nvmlDeviceGetHandleByPciBusId_v2(ctypes.c_char_p(bus), ctypes.byref(h)) == 0
        except AttributeError:
            pass
        if not found:
            found = nv.nvmlDeviceGetHandleByIndex_v2(ctypes.c_uint(torch_index), ctypes.byref(h)) == 0
        if not found:
            raise RuntimeError("no NVML handle")
        self._nvml, self._h = nv, h
        self._reasons_fn = getattr(nv, "nvmlDeviceGetCurrentClocksEventReasons", None) or \
            nv.nvmlDeviceGetCurrentClocksThrottleReasons
        mx = ctypes.c_uint()
        nv.nvmlDeviceGetMaxClockInfo(h, 1, ctypes.byref(mx))
        self.max_mhz = float(mx.value)
        self.source = "nvml"

    def _loop(self):
        nv, h = self._nvml, self._h
        mhz, mw, rs = ctypes.c_uint(), ctypes.c_uint(), ctypes.c_ulonglong()
        while not self._stop.is_set():
            t = time.time()
            if nv.nvmlDeviceGetClockInfo(h, 1, ctypes.byref(mhz)) == 0:
                nv.nvmlDeviceGetPowerUsage(h, ctypes.byref(mw))
                self._reasons_fn(h, ctypes.byref(rs))
                self.samples.append((t, float(mhz.value), mw.value / 1000.0, int(rs.value)))
            self._stop.wait(self.period)

    def start(self):
        if self._nvml is not None:
            self._thread = threading.Thread(target=self._loop, daemon=True)
            self._thread.start()

    def stop(self):
        self._stop.set()
        if self._thread is not None:
            self._thread.join(timeout=2)

    def summary(self, regions) -> dict:
        inside = [s for s in self.samples if any(a <= s[0] <= b for a, b in regions)]
        if not inside:
            return {"sm_mhz": None, "sm_max_mhz": getattr(self, "max_mhz", None), "reasons": ["no samples"],
                    "samples": 0, "source": self.source}
        reasons = sorted({name for s in inside for bit, name in self._REASONS.items() if s[3] & bit})
        return {"sm_mhz": float(np.median([s[1] for s in inside])), "sm_max_mhz": self.max_mhz,
                "reasons": reasons, "samples": len(inside), "power_w_max": round(max(s[2] for s in inside), 1),
                "period_ms": self.period * 1e3, "source": self.source}


def _profiled_traffic(table: dict, source: str, key=None):
    import hashlib

    with open(os.path.join(ROOT, "paper_2607_10661_gb300", "csrc", source), "rb") as f:
        h = hashlib.sha256(f.read()).hexdigest()[:16]
    return table.get(h if key is None else (key, h))


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


def _peaks():
    try:
        with open(MEASURED_PEAKS) as f:
            m = json.load(f)
        return float(m["hbm_gbs"]), float(m["bf16_tflops_sustained"]), "measured"
    except Exception:
        return FALLBACK_HBM_GBS, FALLBACK_BF16_TFLOPS_SUSTAINED, "fallback"


class Regions:
    """Repeats a timed region (K steps) until MIN_REGION_WALL_S of wall time has passed
    (at least three times) and keeps every region's device time and wall interval."""

    def __init__(self, dist, device):
        self.dist, self.device = dist, device
        self.ms, self.walls = [], []

    def run(self, region, min_wall_s=MIN_REGION_WALL_S, min_reps=3):
        import torch

        t_start = time.time()
        while len(self.ms) < min_reps or time.time() - t_start < min_wall_s:
            if self.dist is not None:
                self.dist.barrier()
            torch.cuda.synchronize()
            w0 = time.time()
            ms = region()
            torch.cuda.synchronize()
            w1 = time.time()
            if self.dist is not None:
                self.dist.barrier()
            self.ms.append(ms)
            self.walls.append((w0, w1))
        return self

    def median(self):
        return float(statistics.median(self.ms))


# ----------------------------------------------------------------------------- GPU arm
def _external_record(ev, stream):
    """Record a timing event as a node of the CUDA graph being captured on `stream` (a plain
    cudaEventRecord during capture only orders streams).  Driver API, read-only on settings."""
    r = _libcuda().cuEventRecordWithFlags(ctypes.c_void_p(ev.cuda_event), ctypes.c_void_p(stream.cuda_stream),
                                         ctypes.c_uint(1))   # CU_EVENT_RECORD_EXTERNAL
    if r != 0:
        raise RuntimeError(f"cuEventRecordWithFlags failed ({r})")


_CUDA = []


def _libcuda():
    if not _CUDA:
        _CUDA.append(ctypes.CDLL("libcuda.so.1"))
    return _CUDA[0]


def _capture(fn):
    """A CUDA graph of fn's launches (fn runs once eagerly on a side stream first)."""
    import torch

    side = torch.cuda.Stream()
    side.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(side):
        fn()
    torch.cuda.current_stream().wait_stream(side)
    torch.cuda.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g):
        fn()
    torch.cuda.synchronize()
    return g


def run_gpu(args, rank: int, world: int, dist):
    import torch

    from paper_2607_10661_gb300 import ptd
    from paper_2607_10661_gb300 import synthetic as syn
    from paper_2607_10661_gb300.harness import DeviceWorkload

    local = int(os.environ.get("LOCAL_RANK", "0"))
    torch.cuda.set_device(local)
    dev = f"cuda:{local}"
    import __graft_entry__

    if rank == 0 or not os.path.exists(ptd.LIB_PATH):
        __graft_entry__.build()
    if dist is not None:
        dist.barrier()
    cfg = syn.CONFIGS[args.workload]
    if args.layers:
        cfg = syn.shrink(cfg, layers=args.layers)
    w = syn.Workload(cfg, 1000 + rank)
    dw = DeviceWorkload(w, device=dev)
    nb = step_bytes(w)
    sampling = args.verify == "sampling"
    extras = args.lm_head or args.draft_update or args.ptd_step or sampling
    if extras and (cfg.batch != 1 or cfg.dtype != "bf16"):
        raise SystemExit("--lm-head / --draft-update / --ptd-step / --verify sampling time one-tree bf16 workloads")
    l2 = int(torch.cuda.get_device_properties(local).L2_cache_size)
    # rotating copies of every buffer: consecutive steps use different copies and the copies
    # together are at least three times the L2 size, so no step finds its inputs in L2
    R = 1 if nb["roofline"] >= 3 * l2 or extras else min(512, -(-3 * l2 // nb["roofline"]))
    copies = [dw] + [dw.clone() for _ in range(R - 1)]
    K = args.steps
    n_graphs = -(-R // K)                     # graph j runs steps j*K .. j*K + K - 1 (mod R)
    plan = [[copies[(j * K + i) % R] for i in range(K)] for j in range(n_graphs)]
    if sampling:
        # Alg. 2 at temperature 1: the uniforms are inputs of the step, like the logits
        gu = torch.Generator(device=dev)
        gu.manual_seed(5000 + rank)
        u_acc = torch.rand(w.n_total, device=dev, generator=gu)
        u_bon = torch.rand(cfg.batch, device=dev, generator=gu)
    if args.lm_head:
        # the LM head feeds top-k from the nodes' hidden states: W [vocab][d_model] bf16 and H
        # [N_tot][d_model] (synthetic, seeded; Llama-3-8B's head is 128256 x 4096)
        d_model = 4096
        gh = torch.Generator(device=dev)
        gh.manual_seed(7000 + rank)
        lm_w = (torch.randn((cfg.vocab, d_model), generator=gh, device=dev) / d_model ** 0.5).to(torch.bfloat16)
        lm_h = torch.randn((w.n_total, d_model), generator=gh, device=dev).to(torch.bfloat16)
        lm_ws = torch.empty(ptd.lm_head_workspace_size(w.n_total, cfg.vocab), dtype=torch.uint8, device=dev)
        lm_evs = []
    if args.ptd_step:
        args.draft_update = True
        # the tree's own (unrotated) K and V of every layer, written by the rotary step into
        # the cache slots the attention reads; the candidate pool the draft tree feeds
        gk = torch.Generator(device=dev)
        gk.manual_seed(6000 + rank)
        tree_k = torch.randn((cfg.layers, w.n_total, cfg.hkv, cfg.d), generator=gk, device=dev).to(dw.tdtype)
        tree_v = torch.randn_like(tree_k)
        pool = ptd.CandidatePool(1 << 20, device=dev)
        ret = [torch.zeros(1, dtype=torch.int32, device=dev),
               torch.empty(ptd.MAX_TREE_NODES, dtype=torch.int32, device=dev),
               torch.empty(ptd.MAX_TREE_NODES, dtype=torch.int32, device=dev)]
        pool_step = [0]
    if args.draft_update:
        # the step's tree as a one-seed draft forest, grown by every node's top-1 (width 4,
        # depth 6: the paper's best setting); the output is the next step's draft tree
        du_cnt = torch.tensor([w.n_total], dtype=torch.int32, device=dev)
        du_out = [torch.empty((1,), dtype=torch.int32, device=dev)] + \
                 [torch.empty((1, ptd.MAX_TREE_NODES), dtype=torch.int32, device=dev) for _ in range(3)] + \
                 [torch.empty((1, w.n_total), dtype=torch.int32, device=dev)]

    attn_kernels = [1]   # kernels of one attention call: 2 when split units are merged after it

    def parts_step(d, ev=None, record=None):
        """One step of copy d through the entry points one by one; `record(event)` around the
        attention when timing it."""
        n = 0
        if args.ptd_step:   # positions C + |pi(v)| - 1, rotary encoding, tree K/V into the cache
            n += ptd.tree_rope_append(d.tree, d.cache, 0, d.q, cfg.hq, tree_k, tree_v, 500000.0, d.dev_status)
        if ev is not None:
            record(ev[0])
        na = d.attention()
        attn_kernels[0] = na
        n += na
        if ev is not None:
            record(ev[1])
        if args.lm_head:
            e2 = None
            if ev is not None:
                e2 = (torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
                e2[0].record()
            n += ptd.lm_head_topk(lm_h, lm_w, cfg.k, d.topk_idx, d.topk_val, lm_ws, d.dev_status)
            if e2 is not None:
                e2[1].record()
                lm_evs.append(e2)
        else:
            n += d.topk()
        if args.draft_update:
            n += ptd.draft_tree_update(du_cnt, d.parents.view(1, -1), d.tokens.view(1, -1), d.topk_idx, 1, 4, 6,
                                       ptd.MAX_TREE_NODES, *du_out, d.dev_status)
        if args.ptd_step:   # the grown draft tree joins the pool; C_X for the next step
            pool_step[0] += 1
            n += pool.merge(pool_step[0], du_out[0], du_out[1][0], du_out[2][0], d.dev_status, max_load=1 << 19)
        if sampling:
            n += ptd.verify_sampling(d.tree, d.tokens, d.logits, 1.0, u_acc, u_bon, d.accepted, d.accept_len,
                                     d.bonus, d.dev_status)
            n += d.compact()
        else:
            n += d.verify_and_compact()
        if args.ptd_step:
            n += pool.retrieve(d.bonus[:1], 4, 6, 64, *ret)
        return n

    def call_step(d):
        """One step of copy d through the one-call entry ptd_tree_verify_step (the current stream)."""
        return ptd.tree_verify_step(d.tree, d.cache, d.bufs)

    launches = [0]

    def k_steps(j, step_fn):
        n = 0
        for d in plan[j]:
            n += step_fn(d)
        launches[0] = n
        return n

    for d in copies:
        d.dev_status.zero_()            # sticky status words: cleared once, read after the run
    sampler = ClockSampler(local)
    sampler.start()
    for i in range(max(args.warmup, R)):
        (parts_step if extras else call_step)(copies[i % R])
    torch.cuda.synchronize()
    bad = [int(d.dev_status.item()) for d in copies if int(d.dev_status.item())]
    assert not bad, ptd.status_string(bad[0])

    # ---- value: K steps through the public one-call entry, captured as CUDA graphs and replayed
    # (so that the host's launch overhead is not in the timed region), repeated, median region
    graph_note = None
    graphs = None
    if not extras:
        try:
            graphs = [_capture(lambda j=j: k_steps(j, call_step)) for j in range(n_graphs)]
        except Exception as e:   # reported; the eager loop then gives the value
            graph_note = f"graph capture failed: {e}"[:200]
            graphs = None
    turn = [0]

    def graph_region():
        j = turn[0] % n_graphs
        turn[0] += 1
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record()
        graphs[j].replay()
        b.record()
        torch.cuda.synchronize()
        return a.elapsed_time(b)

    def eager_region():
        j = turn[0] % n_graphs
        turn[0] += 1
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record()
        k_steps(j, parts_step if extras else call_step)
        b.record()
        torch.cuda.synchronize()
        return a.elapsed_time(b)

    main = Regions(dist, dev).run(graph_region if graphs is not None else eager_region)
    launches_per_region = launches[0]   # the kernels of K steps (the captured steps, or the eager ones)
    eager = Regions(dist, dev).run(eager_region) if graphs is not None else main
    status = 0
    for d in copies:
        status |= int(d.dev_status.item())

    # ---- roofline: the same steps through the entry points one by one with timing events
    # around every attention launch (graph nodes when captured), repeated the same way
    attn_pairs = []
    parts_graphs, parts_events = None, None
    if not extras:
        try:
            parts_events = []
            for j in range(n_graphs):
                evs = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(K)]
                for e in evs:          # create the events before the capture
                    e[0].record()
                    e[1].record()
                parts_events.append(evs)
            torch.cuda.synchronize()

            def parts_k(j):
                evs = iter(parts_events[j])
                capturing = torch.cuda.is_current_stream_capturing()
                rec = ((lambda e: _external_record(e, torch.cuda.current_stream())) if capturing else
                       (lambda e: e.record()))
                for d in plan[j]:
                    parts_step(d, next(evs), rec)

            parts_graphs = [_capture(lambda j=j: parts_k(j)) for j in range(n_graphs)]
        except Exception as e:
            graph_note = (graph_note or "") + f" parts graph capture failed: {e}"[:200]
            parts_graphs = None

    def parts_region():
        j = turn[0] % n_graphs
        turn[0] += 1
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        if parts_graphs is not None:
            a.record()
            parts_graphs[j].replay()
            b.record()
            torch.cuda.synchronize()
            attn_pairs.extend(x.elapsed_time(y) for x, y in parts_events[j])
        else:
            evs = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(K)]
            a.record()
            for d, ev in zip(plan[j], evs):
                parts_step(d, ev, lambda e: e.record())
            b.record()
            torch.cuda.synchronize()
            attn_pairs.extend(x.elapsed_time(y) for x, y in evs)
        return a.elapsed_time(b)

    parts = Regions(dist, dev).run(parts_region)
    attn_ms = float(np.mean(attn_pairs))

    # ---- the attention alone, K launches back to back on the stream (each placed by
    # programmatic dependent launch while the one before drains): the roofline's second
    # reading, with no timing event between launches
    b2b_ms = float("nan")
    if not extras:
        def b2b_region():
            j = turn[0] % n_graphs
            turn[0] += 1
            a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            a.record()
            for d in plan[j]:
                d.attention()
            b.record()
            torch.cuda.synchronize()
            return a.elapsed_time(b)

        b2b_ms = Regions(dist, dev).run(b2b_region).median() / K
    lm_ms = float(np.mean([a.elapsed_time(b) for a, b in lm_evs])) if args.lm_head else None
    for d in copies:
        status |= int(d.dev_status.item())

    # ---- end to end: pinned host inputs and outputs through the pipelined host-buffer API
    e2e = None
    if not args.no_e2e and not extras:
        e2e = run_e2e(args, dw, w, dist, dev, torch.cuda.current_stream(), K)

    clocks = sampler.summary(main.walls + parts.walls + (e2e.pop("_walls") if e2e else []))
    sampler.stop()

    ms_main, ms_eager, ms_parts = main.median(), eager.median(), parts.median()
    ms_main, ms_eager, ms_parts, attn_ms, b2b_ms = reduce_over_ranks(
        dist, [ms_main, ms_eager, ms_parts, attn_ms, b2b_ms], dev)
    hbm_peak, tf_peak, peak_kind = _peaks()
    ms_step = ms_main / K
    value = aggregate_rate(world, K, ms_main)
    flops = attention_flops(w)
    achieved_gbs = nb["attention"] / (attn_ms * 1e-3) / 1e9
    achieved_tf = flops / (attn_ms * 1e-3) / 1e12
    tensor_bound = flops / nb["attention"] > 1e12 * tf_peak / (1e9 * hbm_peak)
    if tensor_bound:
        roof = {"bound": "tensor", "achieved": round(achieved_tf, 1), "peak": tf_peak, "unit": "TFLOP/s",
                "frac": round(achieved_tf / tf_peak, 4), "peak_kind": f"{peak_kind} (bf16, sustained)",
                "hbm_achieved_gbs": round(achieved_gbs, 1), "hbm_frac": round(achieved_gbs / hbm_peak, 4)}
    else:
        roof = {"bound": "hbm", "achieved": round(achieved_gbs, 1), "peak": hbm_peak, "unit": "GB/s",
                "frac": round(achieved_gbs / hbm_peak, 4), "peak_kind": peak_kind,
                "tensor_tflops": round(achieved_tf, 1), "tensor_frac": round(achieved_tf / tf_peak, 4)}
    kernel = "tree_attn_tc_kernel" if cfg.dtype == "bf16" else "tree_attn_simt_kernel"
    if attn_kernels[0] == 2:   # timed from the attention's start to the end of the merge of split units
        kernel += " + tree_attn_merge_kernel"
    roof.update({"kernel": kernel, "traffic": _profiled_traffic(PROFILED_ATTENTION_TRAFFIC, "attention_tc.cu",
                                                                 (cfg.name, cfg.layers)),
                 "bytes_per_launch": nb["attention"], "flops_per_launch": flops, "avg_launch_ms": round(attn_ms, 5),
                 "launches_timed": len(attn_pairs),
                 "timing": ("CUDA events recorded as graph nodes around every attention launch of the replayed "
                            "parts loop" if parts_graphs is not None else
                            "CUDA events around every attention launch of the eager parts loop")})
    if b2b_ms == b2b_ms:   # the back-to-back reading (not NaN)
        b2b_frac = ((flops / (b2b_ms * 1e-3) / 1e12) / tf_peak if tensor_bound else
                    (nb["attention"] / (b2b_ms * 1e-3) / 1e9) / hbm_peak)
        roof.update({"avg_launch_ms_back_to_back": round(b2b_ms, 5), "frac_back_to_back": round(b2b_frac, 4),
                     "back_to_back_timing": f"{K} attention calls launched from the host back to back between "
                                            "two CUDA events, divided by the launch count; median of the regions "
                                            "(host-bound where a launch is shorter than the host's call)"})
    l2_note = (f"inputs larger than L2 ({nb['roofline'] / 1e9:.2f} GB read per step vs {l2 >> 20} MB L2)" if R == 1
               else f"{R} copies of every input rotated step by step ({R * nb['roofline'] / 1e6:.0f} MB in all vs "
                    f"{l2 >> 20} MB L2): no step finds its inputs in L2")
    extra_cfg = {
        "verify": "sampling (Alg. 2, temperature 1)" if sampling else "greedy",
        "draft_update": "top-1 expansion, width 4, depth 6 (Alg. 1 step 3)" if args.draft_update else None,
        "top_k_source": ("LM head from hidden states (logits not written)" if args.lm_head else "resident logits"),
        "step_tail": None if sampling else STEP_TAILS[ptd.step_tail(dw.tree, dw.cache, dw.bufs)],
        "ptd_step": ("tree positions + rotary encoding + K/V append, attention, top-k, verification + compaction, "
                     "draft update, pool merge, pool retrieval") if args.ptd_step else None,
        "parallelism": f"replicas x{world}" if world > 1 else "single GPU", "l2": l2_note}
    out = {
        "metric": METRIC,
        "value": round(value, 3),
        "unit": "steps/s",
        "n_gpus": world,
        "steps": K,
        "warmup": args.warmup,
        "ms_per_step": round(ms_step, 5),
        "higher_is_better": True,
        "scaling": "weak",
        "vs_baseline": None,
        "dtype": cfg.dtype,
        "data": "synthetic (seeded N(0,1) Q/K/V, N(0,sigma) logits with a planted boosted token, random pruned trees)",
        "config": bench_config(w, extra_cfg),
        "api": ("entry points one by one (extra parts of the PTD step), eager" if extras else
                "ptd_tree_verify_step (one call per step, device buffers), K steps captured in one CUDA graph and "
                "replayed"),
        "graph_note": graph_note,
        "regions": {"count": len(main.ms), "ms_median": round(ms_main, 4), "ms_min": round(min(main.ms), 4),
                    "ms_max": round(max(main.ms), 4)},
        "eager": {"value": round(aggregate_rate(world, K, ms_eager), 3), "unit": "steps/s",
                  "api": "the same steps called from Python one by one (host launch overhead included)"},
        "step_roofline_bytes": nb["roofline"],
        "hbm_gbs": round(nb["roofline"] / (ms_step * 1e-3) / 1e9, 1),
        "hbm_frac_of_8tbs": round(nb["roofline"] / (ms_step * 1e-3) / 1e9 / NOMINAL_HBM_GBS, 4),
        "hbm_frac_of_measured": round(nb["roofline"] / (ms_step * 1e-3) / 1e9 / hbm_peak, 4),
        "roofline": roof,
        "parts": {"value": round(aggregate_rate(world, K, ms_parts), 3), "unit": "steps/s",
                  "api": "ptd_tree_attention, ptd_topk_draft, ptd_verify_and_compact called one by one with timing "
                         "events around every attention launch (the roofline's timing)",
                  "regions": len(parts.ms),
                  "step_minus_attention_us": round((ms_parts / K - attn_ms) * 1e3, 2)},
        "clocks": clocks,
        "e2e": e2e,
        "lm_head": ({"kernel": "lm_head_topk_kernel", "avg_launch_ms": round(lm_ms, 5),
                     "bytes_per_launch": int(lm_w.numel() * 2 + lm_h.numel() * 2),
                     "achieved_gbs": round((lm_w.numel() * 2 + lm_h.numel() * 2) / (lm_ms * 1e-3) / 1e9, 1),
                     "frac": round((lm_w.numel() * 2 + lm_h.numel() * 2) / (lm_ms * 1e-3) / 1e9 / hbm_peak, 4),
                     "peak_kind": peak_kind,
                     "traffic": (_profiled_traffic(PROFILED_LM_HEAD_TRAFFIC, "lm_head.cu")
                                 if cfg.vocab == 128256 else None),
                     "note": "two launches: the product with per-CTA top-k, then the per-row merge"}
                    if args.lm_head else None),
        "gpu_launches": int(launches_per_region),
        "status": ptd.status_string(status),
    }
    if rank == 0 and not args.no_cpu_baseline:
        out["cpu_baseline"] = cpu_baseline(args.workload, args.cpu_seconds, w.seed)
    return out


def run_e2e(args, dw, w, dist, dev, stream, K):
    """Pipelined host-buffer steps (ptd_pipeline_*), K per region, repeated; the one-step
    host call (a synchronize per step) beside it for contiguous caches."""
    import torch

    from paper_2607_10661_gb300 import ptd

    cfg = w.cfg
    pin = lambda t: t.contiguous().pin_memory()
    tk, tv = dw.tree_rows()
    io_t = dict(q_h=pin(dw.q.cpu()), logits_h=pin(dw.logits.cpu()), tokens_h=pin(dw.tokens.cpu()),
                parents_h=pin(dw.parents.cpu()), node_offsets_h=pin(dw.node_offsets.cpu()),
                ctx_lens_h=pin(dw.ctx_lens.cpu()), tree_k_h=pin(tk.cpu()), tree_v_h=pin(tv.cpu()),
                topk_idx_h=pin(torch.zeros((w.n_total, cfg.k), dtype=torch.int32)),
                topk_val_h=pin(torch.zeros((w.n_total, cfg.k), dtype=torch.float32)),
                accepted_h=pin(torch.zeros((cfg.batch, w.max_nodes), dtype=torch.int32)),
                accept_len_h=pin(torch.zeros(cfg.batch, dtype=torch.int32)),
                bonus_h=pin(torch.zeros(cfg.batch, dtype=torch.int32)),
                new_ctx_h=pin(torch.zeros(cfg.batch, dtype=torch.int32)),
                status_h=pin(torch.zeros(1, dtype=torch.int32)))
    del tk, tv
    outs = ("topk_idx_h", "topk_val_h", "accepted_h", "accept_len_h", "bonus_h", "new_ctx_h", "status_h")
    h2d = sum(io_t[n].numel() * io_t[n].element_size() for n in io_t if n not in outs)
    d2h = sum(io_t[n].numel() * io_t[n].element_size() for n in outs)
    walls = []

    one_step = None
    if not cfg.page_size:
        io = ptd.HostIO(**io_t)

        def host_region():
            a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            a.record(stream)
            for _ in range(K):
                ptd.tree_verify_step_host(dw.tree, dw.cache, dw.bufs, io)
                stream.synchronize()           # the host reads the step's result before the next step
            b.record(stream)
            torch.cuda.synchronize()
            return a.elapsed_time(b)

        for _ in range(3):
            ptd.tree_verify_step_host(dw.tree, dw.cache, dw.bufs, io)
            stream.synchronize()
        r = Regions(dist, dev).run(host_region)
        walls += r.walls
        one_step = (r.median(), int(io_t["status_h"][0]) == 0)

    tree_b, bufs_b = dw.twin_step_buffers()
    es = dw.k.element_size()
    staging = [torch.empty(2 * cfg.layers * w.n_total * cfg.hkv * cfg.d * es, dtype=torch.uint8, device=dev)
               for _ in range(2)]
    pipe = ptd.Pipeline(dw.cache, (dw.tree, tree_b), (dw.bufs, bufs_b), staging)
    io_t2 = {k: (pin(v.clone()) if k in outs else v) for k, v in io_t.items()}
    ios, outs_t = [ptd.HostIO(**io_t), ptd.HostIO(**io_t2)], [io_t, io_t2]
    ok = [True]

    def run_pipeline(n):
        prev = None
        for i in range(n):
            tk_ = pipe.submit(ios[i & 1])
            if prev is not None:
                pipe.wait(prev)
                ok[0] = ok[0] and int(outs_t[(i - 1) & 1]["status_h"][0]) == 0
            prev = tk_
        pipe.wait(prev)
        ok[0] = ok[0] and int(outs_t[(n - 1) & 1]["status_h"][0]) == 0

    def pipe_region():
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record(stream)
        run_pipeline(K)
        b.record(stream)
        torch.cuda.synchronize()
        return a.elapsed_time(b)

    run_pipeline(4)
    r = Regions(dist, dev).run(pipe_region)
    walls += r.walls
    pipe.close()
    world = dist.get_world_size() if dist is not None else 1
    ms_pipe, ms_one = reduce_over_ranks(dist, [r.median(), one_step[0] if one_step else 0.0], dev)
    return {"value": round(aggregate_rate(world, K, ms_pipe), 3), "unit": "steps/s", "steps": K,
            "regions": len(r.ms), "h2d_bytes_per_step": int(h2d), "d2h_bytes_per_step": int(d2h),
            "status_ok": ok[0] and (one_step is None or one_step[1]), "verify": "greedy",
            "api": "ptd_pipeline_submit / ptd_pipeline_wait (uploads and downloads overlapped with compute, two "
                   "steps in flight); every step's inputs uploaded from pinned host memory and its result read by "
                   "the host",
            "one_step_call_value": (round(aggregate_rate(world, K, ms_one), 3) if one_step else None),
            "_walls": walls}


# ----------------------------------------------------------------------------- CPU oracle
def _oracle_worker(conn, name, seed, units, rows):
    """One host process of the oracle step: its share of the attention units (layer, tree,
    KV head) and top-k rows, and the compaction of its units' K and V slices."""
    import oracle
    from paper_2607_10661_gb300 import synthetic as syn

    try:
        cfg = syn.CONFIGS[name]
        w = syn.Workload(cfg, seed)
        G = cfg.hq // cfg.hkv
        data = {}
        for l in sorted({u[0] for u in units}):
            q = syn.widen(w.q_layer(l), cfg.dtype)
            kc, vc = (syn.widen(x, cfg.dtype) for x in w.kv_layer(l))
            for (ll, b, h) in units:
                if ll == l:
                    sl = w.nodes_of(b)
                    data[(l, b, h)] = (np.ascontiguousarray(q[sl][:, h * G:(h + 1) * G]),
                                       np.ascontiguousarray(w.seq_view(kc, b)[:, h:h + 1]),
                                       np.ascontiguousarray(w.seq_view(vc, b)[:, h:h + 1]))
            del q, kc, vc
        lg = syn.widen(w.logits[rows[0]:rows[1]], cfg.dtype)
        conn.send("ready")
        keys = list(data)
        while True:
            msg = conn.recv()
            if msg[0] == "stop":
                break
            if msg[0] == "attention":          # ("attention", m, j): the units u with u % m == j
                m, j = msg[1], msg[2]
                for u in keys[j::m]:
                    q, k, v = data[u]
                    oracle.tree_attention(q, k, v, w.trees[u[1]], int(w.ctx_lens[u[1]]))
                conn.send(None)
            elif msg[0] == "topk":
                idx = np.array([oracle.topk(lg[r], cfg.k)[0] for r in range(len(lg))], np.int32).reshape(-1, cfg.k)
                conn.send(idx)
            elif msg[0] == "compact":          # ("compact", paths, m, j)
                paths, m, j = msg[1], msg[2], msg[3]
                for u in keys[j::m]:
                    q, k, v = data[u]
                    oracle.kv_compact(k, paths[u[1]], int(w.ctx_lens[u[1]]))
                    oracle.kv_compact(v, paths[u[1]], int(w.ctx_lens[u[1]]))
                conn.send(None)
    except Exception as e:  # reported by the parent
        conn.send(("error", repr(e)[-300:]))


def host_cores() -> int:
    try:
        return len(os.sched_getaffinity(0))
    except AttributeError:
        return os.cpu_count() or 1


class OracleStep:
    """Whole oracle steps over the host cores: worker processes (started with spawn, BLAS
    pinned to one thread each) hold contiguous shares of the attention units and top-k rows;
    per step, every worker runs its attention units and top-k rows, the parent verifies
    every tree on this step's greedy targets (top-k column 0), then every worker compacts
    its units' K and V slices along the accepted paths."""

    def __init__(self, name: str, seed: int, cores: int):
        import multiprocessing as mp

        from paper_2607_10661_gb300 import synthetic as syn

        self.w = syn.Workload(syn.CONFIGS[name], seed)
        c = self.w.cfg
        units = [(l, b, h) for l in range(c.layers) for b in range(c.batch) for h in range(c.hkv)]
        self.workers = max(1, min(cores, len(units)))
        n = self.w.n_total
        ctx = mp.get_context("spawn")
        saved = {k: os.environ.get(k) for k in ("OMP_NUM_THREADS", "OPENBLAS_NUM_THREADS", "MKL_NUM_THREADS",
                                                 "CUDA_VISIBLE_DEVICES")}
        os.environ.update(OMP_NUM_THREADS="1", OPENBLAS_NUM_THREADS="1", MKL_NUM_THREADS="1",
                          CUDA_VISIBLE_DEVICES="")
        self.procs, self.conns = [], []
        try:
            for i in range(self.workers):
                u = units[i * len(units) // self.workers:(i + 1) * len(units) // self.workers]
                rows = (i * n // self.workers, (i + 1) * n // self.workers)
                a, b = ctx.Pipe()
                p = ctx.Process(target=_oracle_worker, args=(b, name, seed, u, rows), daemon=True)
                p.start()
                self.procs.append(p)
                self.conns.append(a)
        finally:
            for k, v in saved.items():
                if v is None:
                    os.environ.pop(k, None)
                else:
                    os.environ[k] = v
        for cn in self.conns:
            self._recv(cn)

    @staticmethod
    def _recv(cn):
        m = cn.recv()
        if isinstance(m, tuple) and len(m) == 2 and m[0] == "error":
            raise RuntimeError(m[1])
        return m

    def _round(self, msg):
        for cn in self.conns:
            cn.send(msg)
        return [self._recv(cn) for cn in self.conns]

    def step(self, m: int = 1, j: int = 0) -> float:
        """One oracle step; returns its wall time in seconds.  With m > 1 only every m-th
        attention unit (offset j) is run and compacted, and those two phases' times are
        scaled by m: an estimate of the whole step from a 1/m sample of its units."""
        import oracle

        w = self.w
        t0 = time.perf_counter()
        self._round(("attention", m, j))
        t1 = time.perf_counter()
        idx = np.concatenate(self._round(("topk",)), axis=0)
        target = idx[:, 0]
        paths = []
        for b, par in enumerate(w.trees):
            sl = w.nodes_of(b)
            paths.append(oracle.verify_greedy(par, w.tokens[sl], target[sl])[0])
        t2 = time.perf_counter()
        self._round(("compact", paths, m, j))
        t3 = time.perf_counter()
        return (t1 - t0) * m + (t2 - t1) + (t3 - t2) * m

    def close(self):
        for cn in self.conns:
            try:
                cn.send(("stop",))
            except Exception:
                pass
        for p in self.procs:
            p.join(timeout=10)
            if p.is_alive():
                p.kill()


SAMPLE_DESC = ("whole steps of the workload: every (layer, tree, KV head) attention unit, every top-k row, the "
               "greedy verification of every tree on the step's own top-k column 0 and the compaction of every "
               "layer's K and V, the units and rows split in contiguous shares over worker processes (BLAS pinned to "
               "one thread each), timed on the wall clock per step")


def cpu_baseline(name: str, budget_s: float, seed: int) -> dict:
    """The oracle as it stands on whole steps of the workload: one warm-up step, then as many
    steps as fit in about budget_s (at least one), over every host core."""
    cores = host_cores()
    try:
        st = OracleStep(name, seed, cores)
        try:
            st.step()
            times, t0 = [], time.time()
            while not times or time.time() - t0 < budget_s:
                times.append(st.step())
        finally:
            st.close()
    except Exception as e:  # reported, never fatal for the GPU line
        return {"value": None, "unit": "steps/s", "cores": cores, "kind": "oracle", "error": str(e)[-300:]}
    return {"value": len(times) / float(sum(times)), "unit": "steps/s", "cores": st.workers, "kind": "oracle",
            "steps": len(times), "seconds_per_step": float(np.mean(times)),
            "sample": f"{len(times)} {SAMPLE_DESC}"}


def run_reference(args):
    """--impl reference: the CPU oracle on the host cores, W untimed and K timed steps of the
    same workload.  Steps are whole when K of them fit in --ref-seconds; otherwise every timed
    step runs the attention and compaction of a 1/m sample of the units (a different sample
    each step) with the top-k and verification whole, and those phases' times are scaled by
    m, which the line states."""
    cores = host_cores()
    try:
        st = OracleStep(args.workload, 1000, cores)
    except Exception as e:
        return {"impl": "reference", "unavailable": "oracle workers failed: " + str(e)[-200:]}
    try:
        warm = [st.step() for _ in range(args.warmup)]
        per = float(np.mean(warm))
        m = max(1, int(np.ceil(per * args.steps / args.ref_seconds)))
        times = [st.step(m, i % m) for i in range(args.steps)]
    finally:
        st.close()
    value = len(times) / float(sum(times))
    sample = (f"{len(times)} {SAMPLE_DESC}" if m == 1 else
              f"{len(times)} steps, each the top-k of every row and the verification of every tree whole, and the "
              f"attention and compaction of every {m}-th (layer, tree, KV head) unit (a different 1/{m} each step) "
              f"with those two phases' wall times multiplied by {m}; otherwise as for " + SAMPLE_DESC)
    return {
        "impl": "reference",
        "metric": METRIC,
        "value": value, "unit": "steps/s", "n_gpus": args.gpus, "steps": len(times), "warmup": args.warmup,
        "ms_per_step": float(np.mean(times)) * 1e3, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "config": bench_config(st.w, None),
        "cpu_baseline": {"value": value, "unit": "steps/s", "cores": st.workers, "kind": "oracle",
                         "steps": len(times), "unit_sample_fraction": 1.0 / m, "sample": sample},
        "e2e": {"value": value, "unit": "steps/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }


def main():
    from paper_2607_10661_gb300 import synthetic as syn

    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=20)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", default="ptd", choices=["ptd", "reference"])
    ap.add_argument("--workload", default=DEFAULT_WORKLOAD, choices=list(syn.CONFIG_ORDER))
    ap.add_argument("--layers", type=int, default=0, help="override the layer count (profiling captures)")
    ap.add_argument("--cpu-seconds", type=float, default=20.0)
    ap.add_argument("--ref-seconds", type=float, default=240.0,
                    help="--impl reference: the most the K timed whole oracle steps may take")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-e2e", action="store_true")
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
