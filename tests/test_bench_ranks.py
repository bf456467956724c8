"""The multi-rank host logic of bench.py on CPU: two gloo ranks, max-over-ranks timing and the
reference arm's rank-0-only rule (the one-GPU step runs as independent replicas)."""
import os
import socket
import sys

import pytest
import torch.distributed as dist
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, q):
    sys.path.insert(0, ROOT)
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        import bench
        got = bench.max_over_ranks(10.0 + 5.0 * rank)
        bench.barrier()
        q.put((rank, got))
    finally:
        dist.destroy_process_group()


def test_max_over_ranks_two_gloo_ranks():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(120)
        assert p.exitcode == 0
    res = dict(q.get(timeout=10) for _ in range(2))
    assert res == {0: 15.0, 1: 15.0}


def test_max_over_ranks_without_group_is_identity():
    sys.path.insert(0, ROOT)
    import bench
    assert bench.max_over_ranks(3.5) == 3.5


def test_reference_arm_runs_on_rank_zero_only(capsys):
    sys.path.insert(0, ROOT)
    import bench
    import synth

    class A:
        steps, warmup = 1, 0
    bench.run_reference(A, synth.WORKLOADS[synth.CFG1], rank=1, world=2)
    assert capsys.readouterr().out == ""


def test_reference_arm_prints_the_contract_line(capsys):
    """Rank 0 of the reference arm times the oracle and prints one JSON line with the contract's
    keys (impl, metric, value, unit, e2e with zero copies, cpu_baseline describing the run)."""
    sys.path.insert(0, ROOT)
    import json
    import bench
    import synth

    class A:
        steps, warmup = 2, 1
    bench.run_reference(A, synth.WORKLOADS[synth.CFG1], rank=0, world=1)
    lines = [l for l in capsys.readouterr().out.splitlines() if l.startswith("{")]
    assert len(lines) == 1
    d = json.loads(lines[0])
    assert d["impl"] == "reference" and d["metric"] == bench.METRIC and d["unit"] == bench.UNIT
    assert d["value"] > 0 and d["steps"] == 2 and d["warmup"] == 1 and d["higher_is_better"] is True
    assert d["e2e"] == {"value": d["value"], "unit": d["unit"], "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}
    assert d["cpu_baseline"]["kind"] == "oracle" and d["cpu_baseline"]["value"] == d["value"]
    assert d["config"]["workload"] == synth.CFG1
    # the same config dict as the GPU arm prints for this workload, so the two lines compare
    assert d["config"] == bench.bench_config(synth.WORKLOADS[synth.CFG1], 1)
