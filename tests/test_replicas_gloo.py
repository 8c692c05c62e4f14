"""bench.py host logic on CPU.  The N > 1 path: two gloo ranks, each an independent
replica of the grouped step's host side (its own plan over its own seeded
workload), the job time taken as the slowest rank's, throughput summed over
ranks.  No data-path collective is involved."""
import os
import socket

import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

import bench
import synth


def _free_port():
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    p = s.getsockname()[1]
    s.close()
    return p


def _worker(rank, world, port, out):
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        from paper_2607_16074_gb300 import jnx as J
        w = synth.make_workload("small")
        w.seed = bench.replica_seed(w.seed, rank)
        inp = synth.make_inputs(w)
        plan = J.jnx_group_plan(w.schemas(), bench.oracle_requests(w), len(w.tenants),
                                w.max_samples, w.max_tokens)
        local_ms = 10.0 + 5.0 * rank           # a stand-in for each rank's timed region
        job_ms = bench.max_over_ranks(local_ms, world)
        tps = bench.job_tokens_per_s(plan.n_tokens, world, 3, job_ms)
        out[rank] = (job_ms, tps, plan.n_tokens, float(inp["targets"][:4].sum()))
    finally:
        dist.destroy_process_group()


def test_two_gloo_replicas_weak_scaling():
    world = 2
    mgr = mp.Manager()
    out = mgr.dict()
    mp.spawn(_worker, args=(world, _free_port(), out), nprocs=world, join=True)
    (ms0, tps0, n0, t0), (ms1, tps1, n1, t1) = out[0], out[1]
    assert ms0 == ms1 == 15.0                  # the slowest rank's time
    assert n0 == n1                            # same shapes on every replica
    assert t0 != t1                            # but each replica's own inputs
    assert tps0 == tps1 == pytest.approx(n0 * 2 * 3 / 0.015)


def test_single_rank_needs_no_process_group():
    assert bench.max_over_ranks(7.5, 1) == 7.5
    assert bench.replica_seed(4, 0) == 4


def test_recorded_traffic_only_for_the_captured_launch_shape():
    # the capture's own shape: the 7B-class group's gate/up launch
    rec = bench.RECORDED_TRAFFIC["llama7b"]
    assert bench.recorded_traffic("llama7b", rec[1]) is not None or rec[0] != bench.gemm_source_hash()
    # any other launch (a tenant subset, another width) has no recorded traffic
    assert bench.recorded_traffic("llama7b", (16672, 4096, 11008)) is None
    assert bench.recorded_traffic("mqa2b", (141000, 2048, 16384)) is None


def test_reference_arm_prints_the_contract_line():
    """`bench.py --impl reference` (the fp64 oracle on the host cores) prints
    one JSON line with the keys the benchmark contract asks of that arm."""
    import json
    import subprocess
    import sys
    r = subprocess.run([sys.executable, "bench.py", "--impl", "reference", "--steps", "1",
                        "--warmup", "1"], capture_output=True, text=True, timeout=600,
                       cwd=os.path.dirname(os.path.dirname(os.path.abspath(__file__))))
    assert r.returncode == 0, r.stderr[-2000:]
    lines = [l for l in r.stdout.splitlines() if l.startswith("{")]
    assert len(lines) == 1
    d = json.loads(lines[0])
    assert d["impl"] == "reference" and d["metric"] == bench.METRIC
    assert d["value"] > 0 and d["steps"] == 1 and d["warmup"] == 1
    # what was timed: one whole tenant through two blocks, scaled to depth
    tm = d["timed"]
    assert tm["blocks"] == 2 and tm["scale"] == 16 and tm["tokens"] > 0
    assert tm["full_depth_ms_per_step"] > d["ms_per_step"]
    cb = d["cpu_baseline"]
    assert cb["kind"] == "oracle" and cb["cores"] >= 1 and cb["sample"] and cb["value"] == d["value"]
    e = d["e2e"]
    assert e["value"] == d["value"] and e["unit"] == d["unit"]
    assert e["h2d_bytes_per_step"] == 0 and e["d2h_bytes_per_step"] == 0


def test_oracle_timing_subset_is_whole_tenants_largest_and_smallest():
    """The CPU baseline times whole tenants: every tenant of the one- and
    six-block workloads; otherwise the two with the most tokens and the two
    with the fewest."""
    import synth
    assert bench.oracle_tenant_subset(synth.make_workload("tiny")) == [0, 1]
    assert bench.oracle_tenant_subset(synth.make_workload("small")) == list(range(8))
    for name in ("mqa2b", "zipf2b", "llama7b"):
        w = synth.make_workload(name)
        v = w.backbone.vision_tokens
        tok = {t: sum(s.length(v) for r in w.requests if r.tenant == t for s in r.samples)
               for t in range(len(w.tenants))}
        sub = bench.oracle_tenant_subset(w)
        assert len(sub) == 4
        rest = [t for t in tok if t not in sub]
        lo = sorted(sub, key=lambda t: (tok[t], t))[:2]
        hi = sorted(sub, key=lambda t: (tok[t], t))[2:]
        assert all(tok[t] >= max(tok[x] for x in lo) for t in rest)
        assert all(tok[t] <= min(tok[x] for x in hi) for t in rest)
