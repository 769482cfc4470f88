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
    assert bench.host_cores() >= 1


def test_reference_arm_under_torchrun_prints_once():
    """`bench.py --impl reference` launched as the driver launches it for N = 2: rank 0 runs the
    oracle and prints one JSON line, the other rank exits 0 without work."""
    port = _free_port()
    cmd = [sys.executable, "-m", "torch.distributed.run", "--nnodes=1", "--nproc-per-node", "2", "--master-addr",
           "127.0.0.1", "--master-port", str(port), os.path.join(ROOT, "bench.py"), "--impl", "reference", "--gpus",
           "2", "--steps", "4", "--warmup", "3", "--workload", "tiny-fp32"]
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
    # the steps and warm-up the driver asked for, whole steps, and the GPU arm's config
    assert d["steps"] == 4 and d["warmup"] == 3 and cb["steps"] == 4 and cb["unit_sample_fraction"] == 1.0
    assert d["ms_per_step"] == pytest.approx(1e3 / d["value"])
    sys.path.insert(0, ROOT)
    import bench
    from paper_2607_10661_gb300 import synthetic as syn

    assert d["config"] == bench.bench_config(syn.Workload(syn.CONFIGS["tiny-fp32"], 1000), None)


def test_oracle_step_runs_whole_and_sampled_steps():
    """The CPU baseline's whole oracle step (worker processes started with spawn): whole steps
    and 1/m unit samples both complete, and the sampled estimate scales the sampled phases."""
    sys.path.insert(0, ROOT)
    import bench

    st = bench.OracleStep("tiny-fp32", 1000, 2)
    try:
        assert st.workers == 2                 # 8 (layer, tree, KV head) units over 2 workers
        assert st.step() > 0
        assert st.step(2, 1) > 0               # every 2nd unit of each share, from offset 1
    finally:
        st.close()
    st = bench.OracleStep("llama2-7b-layer", 1000, 3)
    try:
        assert st.workers == 3
        assert st.step() > 0 and st.step(4, 0) > 0
    finally:
        st.close()


def test_clock_summary_keeps_only_samples_inside_the_regions():
    sys.path.insert(0, ROOT)
    import bench

    cs = bench.ClockSampler.__new__(bench.ClockSampler)
    cs.samples = [(1.0, 2070.0, 900.0, 0), (2.0, 1500.0, 1400.0, 0x4), (3.0, 1800.0, 1000.0, 0x40)]
    cs.max_mhz, cs.source, cs.period = 2070.0, "test", 0.01
    s = cs.summary([(1.5, 2.5)])
    assert s["samples"] == 1 and s["sm_mhz"] == 1500.0 and s["reasons"] == ["sw_power_cap"]
    s = cs.summary([(0.5, 1.5), (2.5, 3.5)])
    assert s["samples"] == 2 and s["reasons"] == ["hw_thermal_slowdown"]
    s = cs.summary([(5.0, 6.0)])
    assert s["samples"] == 0 and s["reasons"] == ["no samples"] and s["sm_mhz"] is None


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
