"""The multi-process path of bench.py on the CPU (gloo, world size 2): the step does not
shard, so N GPUs run N independent replicas; what crosses ranks is the timing protocol (the
slowest rank's times, every rank's steps in the whole-job rate) and, for the reference arm,
that rank 0 alone runs and prints while the others exit 0."""
import json
import os
import socket
import subprocess
import sys

import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, q):
    sys.path.insert(0, ROOT)
    import bench

    dist.init_process_group("gloo", init_method=f"tcp://127.0.0.1:{port}", rank=rank, world_size=world)
    try:
        dist.barrier()
        # each rank's own timings: rank 1 is the slow one for the first, rank 0 for the second
        mine = [10.0 + 5.0 * rank, 20.0 - 3.0 * rank, 7.0]
        got = bench.reduce_over_ranks(dist, mine)
        dist.barrier()
        q.put((rank, got, bench.aggregate_rate(world, 100, got[0])))
    finally:
        dist.destroy_process_group()


def test_timing_protocol_over_two_gloo_ranks():
    world, port = 2, _free_port()
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    procs = [ctx.Process(target=_rank_main, args=(r, world, port, q)) for r in range(world)]
    for p in procs:
        p.start()
    out = [q.get(timeout=120) for _ in range(world)]
    for p in procs:
        p.join(timeout=120)
        assert p.exitcode == 0
    for rank, got, rate in out:
        assert got == [15.0, 20.0, 7.0]            # the maximum over the ranks, on every rank
        assert rate == pytest.approx(2 * 100 / 15e-3)   # both replicas' steps over the slowest time
    assert sorted(r for r, _, _ in out) == [0, 1]


def test_single_process_reduction_is_identity():
    sys.path.insert(0, ROOT)
    import bench

    assert bench.reduce_over_ranks(None, [1, 2.5]) == [1.0, 2.5]
    assert bench.aggregate_rate(1, 50, 20.0) == pytest.approx(2500.0)
    # processes running the oracle at once add their rates: two at 2 s and 4 s per step
    assert bench.oracle_rate([[2.0, 2.0], [4.0]]) == pytest.approx(0.5 + 0.25)
    assert bench.host_cores() >= 1


def test_reference_arm_under_torchrun_prints_once():
    """`bench.py --impl reference` launched as the driver launches it for N = 2: rank 0 runs the
    oracle and prints one JSON line, the other rank exits 0 without work."""
    port = _free_port()
    cmd = [sys.executable, "-m", "torch.distributed.run", "--nnodes=1", "--nproc-per-node", "2", "--master-addr",
           "127.0.0.1", "--master-port", str(port), os.path.join(ROOT, "bench.py"), "--impl", "reference", "--gpus",
           "2", "--steps", "2", "--warmup", "1", "--ref-seconds", "5"]
    r = subprocess.run(cmd, cwd=ROOT, capture_output=True, text=True, timeout=300,
                       env=dict(os.environ, CUDA_VISIBLE_DEVICES="", OMP_NUM_THREADS="1"))
    assert r.returncode == 0, r.stderr[-2000:]
    lines = [l for l in r.stdout.splitlines() if l.startswith("{")]
    assert len(lines) == 1
    d = json.loads(lines[0])
    assert d["impl"] == "reference" and d["value"] > 0 and d["n_gpus"] == 2 and d["unit"] == "steps/s"
    cb = d["cpu_baseline"]
    assert cb["kind"] == "oracle" and cb["cores"] >= 1 and cb["value"] == d["value"]
    assert d["e2e"] == {"value": d["value"], "unit": "steps/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}


def test_bench_algorithmic_bytes_and_flops_closed_forms():
    """The roofline numerator of the benchmark's workload from its definition: K and V of
    32 layers x 8 KV heads x (8192 context + 63 tree slots) x 128 x 2 B, Q read and O written
    (32 x 63 x 32 heads x 128 x 2 B each), logits 63 x 128256 x 2 B; attention FLOPs
    4 D Hq L per visible key, a node seeing the context and its own ancestors."""
    import numpy as np

    import bench
    from paper_2607_10661_gb300 import synthetic as syn

    w = syn.Workload(syn.CONFIGS["llama3-8b-gqa"], 1000)
    nb = bench.step_bytes(w)
    assert nb["kv"] == 32 * 8 * (8192 + 63) * 128 * 2 * 2
    assert nb["qo"] == 2 * 32 * 63 * 32 * 128 * 2
    assert nb["logits"] == 63 * 128256 * 2
    assert nb["attention"] == 1115029504 and nb["roofline"] == nb["kv"] + nb["logits"]
    par = w.trees[0]
    depth = [0] * len(par)
    for i in range(1, len(par)):
        depth[i] = depth[par[i]] + 1
    visible = sum(8192 + d + 1 for d in depth)
    assert bench.attention_flops(w) == 4.0 * 128 * 32 * 32 * visible
    assert 2.6e11 < bench.attention_flops(w) < 2.8e11   # 272.7 GFLOP per step
    assert np.isclose(nb["attention"] / 1e6, 1115.0, atol=0.1)
