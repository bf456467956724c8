"""Dynamic Partitioning (Section 4.1, Algorithm 1), Eq. 2 and Eq. 3 - oracle, fp64, pure Python.

Test infrastructure only (see oracle/__init__.py).

Algorithm 1 estimates each worker's compute power, normalises it, and sizes the
next partition as |D^m_{t+1}| = CP_m * |D|.  The paper leaves the integer
rounding of that product open; the reading used here (and mirrored bit for bit
by the library's host rule) is:

1. S = sum_m c_m, summed left to right in fp64.
2. q_m = (c_m / S) * N, in exactly that operation order (normalise, Alg. 1,
   then multiply by |D|).
3. f_m = floor(q_m); R = N - sum_m f_m.
4. The R workers with the largest remainders r_m = q_m - f_m get one more
   sample; equal remainders go to the lower worker index (largest-remainder /
   Hamilton rounding: sum n = N and |n_m - q_m| < 1).
5. Every worker keeps at least one sample: for each m in increasing order with
   n_m = 0, one sample moves from the worker with the largest n (ties to the
   lower index).  A worker with zero samples has no mean loss under Eq. 1.
6. Samples are assigned in contiguous blocks in worker order:
   seg_m = [off_m, off_m + n_m), off = exclusive prefix sum of n.

At t = 0 (Algorithm 1, first branch) every CP is equal: the even split.
"""
from __future__ import annotations

import math
from typing import List, Sequence


def compute_power(sizes: Sequence[float], times: Sequence[float]) -> List[float]:
    """Eq. 2: CP_m = |D_m| / X_m (samples per second)."""
    return [float(d) / float(x) for d, x in zip(sizes, times)]


def predicted_times(sizes: Sequence[float], cp: Sequence[float]) -> List[float]:
    """Eq. 3: X'_m = |D'_m| / CP_m."""
    return [float(d) / float(c) for d, c in zip(sizes, cp)]


def _validate(cp: Sequence[float], n: int) -> None:
    m = len(cp)
    if m < 1:
        raise ValueError("need at least one worker")
    if n < m:
        raise ValueError(f"global batch {n} smaller than worker count {m}")
    for c in cp:
        if not (isinstance(c, (int, float)) and math.isfinite(c) and c > 0.0):
            raise ValueError(f"compute power must be finite and > 0, got {c!r}")


def quotas(cp: Sequence[float], n: int) -> List[float]:
    """Algorithm 1: normalise the CPs, then multiply by |D|."""
    s = 0.0
    for c in cp:
        s = s + float(c)
    return [(float(c) / s) * float(n) for c in cp]


def partition_sizes(cp: Sequence[float], n: int) -> List[int]:
    """Integer partition sizes n_m for compute powers cp over a batch of n samples."""
    cp = [float(c) for c in cp]
    _validate(cp, n)
    m = len(cp)
    q = quotas(cp, n)
    f = [math.floor(v) for v in q]
    rem = [q[i] - f[i] for i in range(m)]
    r = n - sum(f)
    if r < 0 or r > m:
        raise ValueError("rounding residue out of range")
    order = sorted(range(m), key=lambda i: (-rem[i], i))
    sizes = list(f)
    for k in range(r):
        sizes[order[k]] += 1
    for i in range(m):
        if sizes[i] == 0:
            donor = max(range(m), key=lambda j: (sizes[j], -j))
            sizes[donor] -= 1
            sizes[i] += 1
    return sizes


def even_sizes(m: int, n: int) -> List[int]:
    """Algorithm 1, t = 0: CP_m = 1/M for every worker."""
    return partition_sizes([1.0] * m, n)


def offsets(sizes: Sequence[int]) -> List[int]:
    off = [0]
    for s in sizes:
        off.append(off[-1] + int(s))
    return off


def index_map(sizes: Sequence[int]) -> List[int]:
    """Sample -> worker: sample i belongs to worker m for off_m <= i < off_{m+1}."""
    out = []
    for m, s in enumerate(sizes):
        out.extend([m] * int(s))
    return out


def dynamic_partitioning(t: int, mean_times: Sequence[float], sizes: Sequence[int], n: int,
                         m: int) -> List[int]:
    """Algorithm 1 as a whole: the sizes of D_{t+1} from the mean batch times X_t of D_t."""
    if t == 0:
        return even_sizes(m, n)
    return partition_sizes(compute_power(sizes, mean_times), n)


class CPHistory:
    """Compute-power estimate from a history of measurements (Section 4.1: the CPs may come from
    the last epoch only, or from a history of epochs).  Reading: mode "last" uses the newest
    measurement; "ema" keeps e = a * c + (1 - a) * e (the first measurement initialises e);
    "window" averages the last k measurements (summed oldest first, then divided by their count).
    fp64, per worker, in exactly these operation orders."""

    def __init__(self, mode: str = "last", param: float = 0.0):
        self.mode, self.param = mode, float(param)
        self.ema = None
        self.window: List[List[float]] = []

    def update(self, cp: Sequence[float]) -> List[float]:
        cp = [float(c) for c in cp]
        if self.mode == "last":
            return cp
        if self.mode == "ema":
            a = self.param
            if self.ema is None:
                self.ema = list(cp)
            else:
                self.ema = [a * c + (1.0 - a) * e for c, e in zip(cp, self.ema)]
            return list(self.ema)
        k = int(self.param)
        self.window.append(cp)
        if len(self.window) > k:
            self.window.pop(0)
        out = []
        for m in range(len(cp)):
            acc = 0.0
            for row in self.window:
                acc = acc + row[m]
            out.append(acc / float(len(self.window)))
        return out
