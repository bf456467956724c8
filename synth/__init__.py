"""Seeded synthetic workloads shared by the CUDA path's tests/bench and the CPU oracle.

This module holds no arithmetic of the method itself (no partition rule, no
forward/backward pass, no synchronisation, no update). It only draws inputs:

* images x ~ N(0, 1) in fp32, shaped like CIFAR10 (3x32x32, flattened for the
  MLPs) or like the wider 4096-feature MLP workload; labels uniform over C
  classes (the paper trains on CIFAR10, Section 5; the dataset itself is not
  used, seeded normals of its shape stand in for it);
* He-normal initial parameters W ~ N(0, 2 / fan_in), biases zero, flat fp32
  vector in the layout [W1, b1, W2, b2, ...] (W row-major [out, in]; conv
  weights [Cout, Cin, 3, 3]);
* per-worker compute weights: fixed ratios, a lognormal draw, or the seeded
  multiplicative random walk that simulates drifting worker speed (the paper
  simulates heterogeneity by slowing a subset of workers, Section 5).

Every array is a pure function of the seed, so the GPU path and the oracle see
byte-identical inputs.
"""
from __future__ import annotations

import dataclasses
from typing import List, Optional, Sequence

import numpy as np

# Architecture tags (mirror the C enum values in include/hs.h).
MLP = 0
CNN = 1

# Fixed CNN topology: (Cout, stride) per 3x3 conv, then global average pool and one FC layer.
CNN_CONVS = ((64, 1), (128, 2), (256, 2))


@dataclasses.dataclass(frozen=True)
class Workload:
    name: str
    arch: int
    dims: tuple            # MLP: (d0, d1, ..., dL); CNN: (Cin, H, W, c1, c2, c3, classes)
    n_classes: int
    global_batch: int
    workers: int
    weights: Optional[tuple]   # static compute weights, or None (drift / lognormal filled in below)
    steps: int
    lr: float
    seed: int = 0
    weight_kind: str = "static"   # "static" | "lognormal" | "drift"
    repartition_every: int = 0     # drift workloads: steps between repartitions

    @property
    def in_features(self) -> int:
        if self.arch == MLP:
            return self.dims[0]
        cin, h, w = self.dims[:3]
        return cin * h * w


def _cnn_dims(cin=3, h=32, w=32, c=(64, 128, 256), classes=10):
    return (cin, h, w, c[0], c[1], c[2], classes)


# The five workloads.  The paper leaves some steps and learning rates open; these are proposed
# readings: the drifting 2048-wide MLP at lr 0.01, the CNN and the 8192-wide MLP at 10 steps and
# lr 0.01.
WORKLOADS = {
    "mlp_3072_256_10_b128_m2": Workload(
        "mlp_3072_256_10_b128_m2", MLP, (3072, 256, 10), 10, 128, 2, (1.0, 3.0), 10, 0.01),
    "mlp_3072_1024x2_10_b1024_m4": Workload(
        "mlp_3072_1024x2_10_b1024_m4", MLP, (3072, 1024, 1024, 10), 10, 1024, 4,
        (1.0, 1.0, 2.0, 4.0), 100, 0.05),
    "mlp_3072_2048x2_10_b4096_m8_drift": Workload(
        "mlp_3072_2048x2_10_b4096_m8_drift", MLP, (3072, 2048, 2048, 10), 10, 4096, 8, None,
        200, 0.01, weight_kind="drift", repartition_every=10),
    "cnn_c64_c128s2_c256s2_b512_m4": Workload(
        "cnn_c64_c128s2_c256s2_b512_m4", CNN, _cnn_dims(), 10, 512, 4, (1.0, 2.0, 3.0, 6.0), 10, 0.01),
    "mlp_4096_8192x2_1000_b16384_m16": Workload(
        "mlp_4096_8192x2_1000_b16384_m16", MLP, (4096, 8192, 8192, 1000), 1000, 16384, 16, None,
        10, 0.01, weight_kind="lognormal"),
}
CFG1, CFG2, CFG3, CFG4, CFG5 = (
    "mlp_3072_256_10_b128_m2", "mlp_3072_1024x2_10_b1024_m4", "mlp_3072_2048x2_10_b4096_m8_drift",
    "cnn_c64_c128s2_c256s2_b512_m4", "mlp_4096_8192x2_1000_b16384_m16")


# ----------------------------------------------------------------------------- parameter layout
def mlp_shapes(dims: Sequence[int]) -> List[tuple]:
    """Shapes in flat order: W1 [d1, d0], b1 [d1], W2 [d2, d1], ..."""
    out = []
    for l in range(1, len(dims)):
        out.append((dims[l], dims[l - 1]))
        out.append((dims[l],))
    return out


def cnn_shapes(dims: Sequence[int]) -> List[tuple]:
    cin, _, _, c1, c2, c3, classes = dims
    out = []
    prev = cin
    for c in (c1, c2, c3):
        out.append((c, prev, 3, 3))
        out.append((c,))
        prev = c
    out.append((classes, prev))
    out.append((classes,))
    return out


def param_shapes(arch: int, dims: Sequence[int]) -> List[tuple]:
    return mlp_shapes(dims) if arch == MLP else cnn_shapes(dims)


def param_count(arch: int, dims: Sequence[int]) -> int:
    return int(sum(int(np.prod(s)) for s in param_shapes(arch, dims)))


# ----------------------------------------------------------------------------- draws
def make_batch(wl: Workload, seed: Optional[int] = None, n: Optional[int] = None):
    """x ~ N(0,1) fp32 [N, features] (CNN: [N, Cin, H, W]), y ~ U{0..C-1} int32 [N]."""
    seed = wl.seed if seed is None else seed
    n = wl.global_batch if n is None else n
    rng = np.random.default_rng(seed)
    if wl.arch == MLP:
        x = rng.standard_normal((n, wl.dims[0]), dtype=np.float32)
    else:
        cin, h, w = wl.dims[:3]
        x = rng.standard_normal((n, cin, h, w), dtype=np.float32)
    y = rng.integers(0, wl.n_classes, n, dtype=np.int32)
    return x, y


def he_normal_params(arch: int, dims: Sequence[int], seed: int) -> np.ndarray:
    """Flat fp32 parameters: every weight tensor N(0, 2/fan_in) in fp32, biases zero."""
    rng = np.random.default_rng(seed)
    parts = []
    for shape in param_shapes(arch, dims):
        if len(shape) == 1:
            parts.append(np.zeros(shape, dtype=np.float32))
        else:
            fan_in = int(np.prod(shape[1:]))
            w = rng.standard_normal(shape, dtype=np.float32)
            w *= np.float32(np.sqrt(2.0 / fan_in))
            parts.append(w.reshape(-1))
    return np.concatenate([p.reshape(-1) for p in parts]).astype(np.float32)


def make_params(wl: Workload, seed: Optional[int] = None) -> np.ndarray:
    seed = (wl.seed if seed is None else seed) + 1
    return he_normal_params(wl.arch, wl.dims, seed)


def lognormal_weights(m: int, seed: int) -> np.ndarray:
    return np.random.default_rng(seed + 3).lognormal(0.0, 0.5, m)


def drift_walk(m: int, steps: int, seed: int, sigma: float = 0.1) -> np.ndarray:
    """Per-worker speed c_m(t), t = 0..steps: c(0) = 1, c(t+1) = c(t) * exp(sigma * z_t)."""
    z = np.random.default_rng(seed + 2).standard_normal((steps, m))
    c = np.ones((steps + 1, m))
    for t in range(steps):
        c[t + 1] = c[t] * np.exp(sigma * z[t])
    return c


def window_throughputs(speeds: np.ndarray) -> np.ndarray:
    """Measured samples/s over a window of steps in which worker m ran n_m samples per step at
    speed c_m(t) (time n_m / c_m(t)): n_m / mean_t(n_m / c_m(t)) = 1 / mean_t(1 / c_m(t))."""
    return 1.0 / np.mean(1.0 / speeds, axis=0)


def initial_weights(wl: Workload, seed: Optional[int] = None) -> np.ndarray:
    seed = wl.seed if seed is None else seed
    if wl.weight_kind == "static":
        return np.asarray(wl.weights, dtype=np.float64)
    if wl.weight_kind == "lognormal":
        return lognormal_weights(wl.workers, seed)
    return np.ones(wl.workers)        # drift: starts even (Algorithm 1, t = 0)
