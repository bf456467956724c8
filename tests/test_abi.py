"""The C ABI without a GPU: the library loads, exports every declared entry point, and its
host-side partition rule (Algorithm 1) is bit-exact with the oracle."""
import ctypes
import json
import math
import os
import re

import numpy as np
import pytest

import synth
import paper_2110_08941_gb300 as hs
from oracle import partition as P

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _declared():
    names = set()
    for f in os.listdir(os.path.join(ROOT, "include")):
        if f.endswith(".h"):
            src = open(os.path.join(ROOT, "include", f)).read()
            src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
            names |= set(re.findall(r"\b(hs_[a-z0-9_]+)\s*\(", src))
    return names


def test_every_declared_symbol_is_exported():
    lib = ctypes.CDLL(hs.LIB_PATH)
    declared = _declared()
    assert {"hs_init", "hs_partition", "hs_step", "hs_destroy", "hs_partition_sizes"} <= declared
    for name in sorted(declared):
        assert hasattr(lib, name), name
    assert set(hs.EXPORTED) == declared


def test_partition_sizes_golden():
    cases = json.load(open(os.path.join(ROOT, "tests", "golden", "partition_examples.json")))["cases"]
    for c in cases:
        assert hs.hs_partition_sizes(c["cp"], c["N"]) == c["sizes"]


def test_partition_sizes_bitexact_random():
    rng = np.random.default_rng(123)
    for it in range(4000):
        m = int(rng.integers(1, 33))
        n = int(rng.integers(m, 70000))
        kind = it % 4
        if kind == 0:
            cp = rng.lognormal(0, 1.0, m)
        elif kind == 1:
            cp = rng.integers(1, 5, m).astype(float)
        elif kind == 2:
            cp = rng.uniform(1e-6, 1.0, m)
        else:
            cp = np.exp(rng.uniform(-30, 30, m))     # wide dynamic range: many workers at the 1-sample floor
        cp = [float(v) for v in cp]
        assert hs.hs_partition_sizes(cp, n) == P.partition_sizes(cp, n), (cp, n)


def test_partition_sizes_workload_weights():
    for name, wl in synth.WORKLOADS.items():
        w = list(synth.initial_weights(wl))
        assert hs.hs_partition_sizes(w, wl.global_batch) == P.partition_sizes(w, wl.global_batch)
    w = synth.drift_walk(8, 200, 0)
    for t in range(10, 201, 10):
        tp = list(synth.window_throughputs(w[t - 10:t]))
        assert hs.hs_partition_sizes(tp, 4096) == P.partition_sizes(tp, 4096)


@pytest.mark.parametrize("cp,n", [([1.0, 1.0], 1), ([1.0, -1.0], 4), ([1.0, 0.0], 4),
                                  ([1.0, math.inf], 4), ([1.0, math.nan], 4), ([1e308, 1e308], 4)])
def test_partition_sizes_rejects(cp, n):
    with pytest.raises(hs.HsError) as e:
        hs.hs_partition_sizes(cp, n)
    assert e.value.status == hs.HS_ERR_INVALID_ARG


def test_param_count():
    assert hs.hs_param_count(hs.HS_MLP, (3072, 256, 10)) == 789258
    assert hs.hs_param_count(hs.HS_MLP, (3072, 1024, 1024, 10)) == 4206602
    assert hs.hs_param_count(hs.HS_MLP, (3072, 2048, 2048, 10)) == 10510346
    assert hs.hs_param_count(hs.HS_MLP, (4096, 8192, 8192, 1000)) == 108872680
    assert hs.hs_param_count(hs.HS_CNN, synth.WORKLOADS[synth.CFG4].dims) == 373386
    for wl in synth.WORKLOADS.values():
        assert hs.hs_param_count(wl.arch, wl.dims) == synth.param_count(wl.arch, wl.dims)


def test_init_rejects_bad_arguments_before_touching_the_gpu():
    with pytest.raises(hs.HsError) as e:
        hs.hs_init(hs.HS_MLP, (16, 8, 4), M=4, global_batch=3)
    assert e.value.status == hs.HS_ERR_INVALID_ARG
    with pytest.raises(hs.HsError) as e:
        hs.hs_init(hs.HS_MLP, (16, 8, 4), M=2, global_batch=8, compute_weights=[1.0, -2.0])
    assert e.value.status == hs.HS_ERR_INVALID_ARG
    with pytest.raises(hs.HsError) as e:
        hs.hs_init(hs.HS_MLP, (16, 8, 4), M=0, global_batch=8)
    assert e.value.status == hs.HS_ERR_INVALID_ARG


def test_status_strings():
    lib = ctypes.CDLL(hs.LIB_PATH)
    lib.hs_status_string.restype = ctypes.c_char_p
    assert lib.hs_status_string(0) == b"HS_OK"
    assert lib.hs_status_string(5) == b"HS_ERR_DEVICE_CHECK"


def test_cosine_lr_matches_oracle():
    from oracle import sgd
    for t in range(0, 120, 7):
        assert hs.hs_cosine_lr(0.1, 0.001, t, 100) == pytest.approx(sgd.cosine_lr(0.1, 0.001, min(t, 100), 100),
                                                                    rel=0, abs=1e-15)
    assert hs.hs_cosine_lr(0.1, 0.0, 5, 0) == 0.1


def test_index_map_outputs_are_checked_before_the_library_is_called(monkeypatch):
    """hs_partition_noalloc writes N int32 through the tensor's pointer: a short, int64, strided
    or host tensor is refused by the binding before any library call (so before any launch)."""
    import torch
    from paper_2110_08941_gb300 import binding

    calls = []

    class Recorder:
        def __getattr__(self, name):
            def f(*a):
                calls.append(name)
                return 0
            return f

    monkeypatch.setattr(binding, "_lib", Recorder())
    bad = [torch.zeros(7, dtype=torch.int32),                       # host memory, right length
           torch.zeros(6, dtype=torch.int32),                       # short
           torch.zeros(7, dtype=torch.int64),                       # wrong element type
           torch.zeros(14, dtype=torch.int32)[::2],                 # not contiguous
           np.zeros(7, dtype=np.int32)]                             # not a tensor
    for t in bad:
        with pytest.raises(ValueError):
            hs.hs_partition_noalloc([1.0, 2.0], 7, t)
    assert calls == []
