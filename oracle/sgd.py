"""Gradient synchronisation and the SGD update - oracle, fp64 NumPy.

Test infrastructure only (see oracle/__init__.py).

* Sync-SGD / DP-SGD (Section 1): g_t = (1/M) sum_m g^m_t.
* EDP-SGD (Section 4.2): each g^m_t is weighted by the worker's normalised
  compute power before the exchange.  Reading: the weights are the realised
  normalised partition sizes w_m = n_m / N (they sum to 1, so the step size
  keeps its scale; they differ from the normalised CP by integer rounding only,
  at most 1/N), and the exchange then sums.  With mean per-worker losses this
  makes g the gradient of the mean loss over the whole global batch.
  The literal alternative (1/M) sum_m CP_m g^m is kept as "cp_literal".
* Update (Section 1): theta_{t+1} = theta_t - eta_t g_t (plain SGD).

The reported loss is sum_m w_m L_m with the same weights, at theta_t.

The training recipe of Section 5 adds, on top of the synchronised gradient g:
* weight decay lambda and momentum mu (heavy ball, no dampening):
  d = g + lambda * theta;  b = d on the first step, b = mu * b + d afterwards;
  theta <- theta - eta_t * b;
* cosine annealing of the learning rate over T steps:
  eta_t = eta_min + (eta_0 - eta_min) * (1 + cos(pi * t / T)) / 2.
"""
from __future__ import annotations

from typing import Callable, Optional, Sequence

import numpy as np

from . import partition as _part

SYNC_MEAN = 0
SYNC_CP_WEIGHTED = 1
SYNC_CP_LITERAL = 2


def sync_weights(sizes: Sequence[int], mode: int, cp: Optional[Sequence[float]] = None) -> np.ndarray:
    m = len(sizes)
    n = float(sum(sizes))
    if mode == SYNC_MEAN:
        return np.full(m, 1.0 / m)
    if mode == SYNC_CP_WEIGHTED:
        return np.array([s / n for s in sizes], dtype=np.float64)
    if mode == SYNC_CP_LITERAL:
        cp = np.asarray(cp, dtype=np.float64)
        return (cp / cp.sum()) / m
    raise ValueError(f"unknown sync mode {mode}")


def worker_grads(grad_fn: Callable, theta, dims, x, y, sizes):
    """[(L_m, g^m)] for each worker's contiguous segment."""
    off = _part.offsets(sizes)
    out = []
    for m in range(len(sizes)):
        sl = slice(off[m], off[m + 1])
        out.append(grad_fn(theta, dims, x[sl], y[sl]))
    return out


def step(grad_fn: Callable, theta, dims, x, y, sizes, lr: float, mode: int,
         keep_slabs: bool = False, cp=None, **grad_kwargs):
    """One synchronous step: per-worker (L_m, g^m), g = sum_m w_m g^m, theta - lr * g.

    Returns (theta_new fp64, loss, g, slabs or None, per-worker losses).  grad_kwargs go to
    grad_fn (e.g. the ReLU-decision precision of the per-worker gradient).
    Accumulates sum_m w_m g^m worker by worker, so memory stays at O(P) unless
    the per-worker gradients are asked for.
    """
    theta = np.asarray(theta, dtype=np.float64)
    w = sync_weights(sizes, mode, cp)
    off = _part.offsets(sizes)
    g = np.zeros_like(theta)
    slabs = [] if keep_slabs else None
    losses = []
    for m in range(len(sizes)):
        sl = slice(off[m], off[m + 1])
        l_m, g_m = grad_fn(theta, dims, x[sl], y[sl], **grad_kwargs)
        losses.append(l_m)
        g += w[m] * g_m
        if keep_slabs:
            slabs.append(g_m)
    loss = float(np.dot(w, np.asarray(losses)))
    return theta - lr * g, loss, g, slabs, losses


def momentum_update(theta, g, buf, lr: float, momentum: float, weight_decay: float):
    """One update of the Section 5 recipe; buf is None on the first step.  Returns (theta, buf)."""
    theta = np.asarray(theta, dtype=np.float64)
    d = np.asarray(g, dtype=np.float64) + weight_decay * theta
    buf = d.copy() if buf is None else momentum * buf + d
    return theta - lr * buf, buf


def cosine_lr(eta0: float, eta_min: float, t: int, T: int) -> float:
    """Cosine annealing (Section 5): eta_min + (eta0 - eta_min) * (1 + cos(pi t / T)) / 2."""
    return eta_min + (eta0 - eta_min) * (1.0 + np.cos(np.pi * t / T)) / 2.0
