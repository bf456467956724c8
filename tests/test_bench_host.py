"""Host-side measurement logic of bench.py: the straggler simulation (Section 3's X_(M)) and the
roofline bookkeeping helpers."""
import os
import sys

import numpy as np

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)

import bench  # noqa: E402
import synth  # noqa: E402
from oracle import partition as P  # noqa: E402


def test_straggler_simulation_matches_oracle_schedule():
    sim = bench.straggler_simulation(seed=0, steps=60, every=10)
    wl = synth.WORKLOADS[synth.CFG3]
    c = synth.drift_walk(wl.workers, 60, 0)
    sizes = P.even_sizes(wl.workers, wl.global_batch)
    t_dp = 0.0
    for t in range(60):
        t_dp += max(sizes[k] / c[t][k] for k in range(wl.workers))
        if (t + 1) % 10 == 0:
            sizes = P.partition_sizes(list(synth.window_throughputs(c[t - 9:t + 1])), wl.global_batch)
    assert sim["sum_max_time_dynamic_partitioning"] == t_dp
    # the ideal split is a lower bound, the even split the Sync-SGD schedule Dynamic Partitioning improves on
    assert sim["sum_time_ideal_split"] <= sim["sum_max_time_dynamic_partitioning"] <= sim["sum_max_time_even"]


def test_first_window_is_even_in_both_schedules():
    one = bench.straggler_simulation(seed=3, steps=10, every=10)
    assert np.isclose(one["sum_max_time_even"], one["sum_max_time_dynamic_partitioning"])


def test_gemm_flops_of_the_headline_workload():
    f = bench.gemm_flops(synth.WORKLOADS[synth.CFG5])
    assert abs(sum(f.values()) - 9.6014e12) / 9.6014e12 < 1e-4
    cnn = bench.gemm_flops(synth.WORKLOADS[synth.CFG4])
    assert abs(sum(cnn.values()) - 1.196e11) / 1.196e11 < 1e-3


def test_heterogeneity_replica_dynamic_partitioning_helps():
    r = bench.heterogeneity_simulation(4e-7, seed=1)
    for level in ("low", "high"):
        assert r[level]["speedup"] > 1.0
        sizes = r[level]["dynamic_partitioning"]["last_sizes"]
        assert sum(sizes) == 8 * 128
        # delayed workers (even index) end with fewer samples than the undelayed ones
        assert max(sizes[0::2]) < min(sizes[1::2])
    assert r["high"]["speedup"] > r["low"]["speedup"]
    assert r == bench.heterogeneity_simulation(4e-7, seed=1)      # seeded, deterministic
