"""Per-worker loss and gradient of the MLP workloads - oracle, fp64 NumPy.

Test infrastructure only (see oracle/__init__.py).

Eq. 1 defines worker m's objective as an expectation over its own data,
f_m(theta) = E_{x ~ D^m} f(theta; x); on a minibatch that is the mean of the
per-sample losses over the worker's segment:

    L_m(theta) = (1 / n_m) * sum_{i in seg_m} CE(z_i, y_i),  CE(z, y) = logsumexp(z) - z_y,

and Section 1 takes g^m_t as the gradient of that local objective.  The model:
A_l = H_{l-1} W_l^T + b_l, H_l = ReLU(A_l) for hidden layers, z = A_L (linear
last layer), H_0 = x.  W_l is [out, in] (row-major), parameters are one flat
vector [W1, b1, W2, b2, ...].  ReLU'(0) is taken as 0.

Back-propagation is written out layer by layer (no autodiff): for the last
layer dL/dA_L = (softmax(z) - onehot(y)) / n_m, and for every layer
dW_l = dA_l^T H_{l-1}, db_l = sum_rows dA_l, dA_{l-1} = (dA_l W_l) * 1[A_{l-1} > 0].
Inputs are the fp32 arrays the GPU path sees, promoted to fp64.

ReLU'(A) = 1[A > 0] is a floating-point value deciding a 0/1.  A kernel with bf16
operands (fp32 accumulation) decides it from its own pre-activation, which sits
within bf16 rounding of the exact one; where |A| is that small the two decisions
differ, and each flip moves a whole entry of the backward signal.  So that both
sides take the decision in the same precision, `decide` (optional) names an
operand rounding: the masks then come from the forward pass evaluated with
rounded operands (H_0 = x, W_l and the stored activations rounded, exact
accumulation), while every value of the loss and gradient stays fp64.  With
`decide=None` the masks come from the fp64 forward itself.
"""
from __future__ import annotations

from typing import List, Sequence, Tuple

import numpy as np


def layout(dims: Sequence[int]) -> Tuple[List[tuple], int]:
    """[(W_offset, (out, in), b_offset, out)] per layer and the total parameter count P."""
    off = 0
    lay = []
    for l in range(1, len(dims)):
        o, i = int(dims[l]), int(dims[l - 1])
        w_off = off
        off += o * i
        b_off = off
        off += o
        lay.append((w_off, (o, i), b_off, o))
    return lay, off


def unpack(theta: np.ndarray, dims: Sequence[int]):
    lay, p = layout(dims)
    assert theta.size == p, (theta.size, p)
    ws, bs = [], []
    for w_off, shape, b_off, o in lay:
        ws.append(theta[w_off:w_off + shape[0] * shape[1]].reshape(shape))
        bs.append(theta[b_off:b_off + o])
    return ws, bs


def forward(theta: np.ndarray, dims: Sequence[int], x: np.ndarray):
    """Pre-activations A_l and activations H_l (H_0 = x); returns (A list, H list)."""
    ws, bs = unpack(np.asarray(theta, dtype=np.float64), dims)
    h = np.asarray(x, dtype=np.float64)
    acts, hs = [], [h]
    n_layers = len(ws)
    for l in range(n_layers):
        a = h @ ws[l].T + bs[l]
        acts.append(a)
        if l < n_layers - 1:
            h = np.maximum(a, 0.0)
            hs.append(h)
    return acts, hs


def round_bf16(a) -> np.ndarray:
    """Round to the nearest bfloat16 (8 significant bits, ties to even), from the fp32 value.

    bfloat16 is the top half of an IEEE fp32 word; round-to-nearest-even on the discarded low
    16 bits is adding 0x7FFF plus the lowest kept bit, then truncating.  Finite inputs only."""
    f = np.ascontiguousarray(np.asarray(a, dtype=np.float32))
    u = f.view(np.uint32).astype(np.uint64)
    kept_lsb = (u >> np.uint64(16)) & np.uint64(1)
    r = ((u + np.uint64(0x7FFF) + kept_lsb) >> np.uint64(16)) << np.uint64(16)
    return r.astype(np.uint32).view(np.float32).astype(np.float64)


def round_fp32(a) -> np.ndarray:
    """Round to the nearest fp32 value (the storage precision of the fp32 check path)."""
    return np.asarray(a, dtype=np.float32).astype(np.float64)


def relu_decisions(theta: np.ndarray, dims: Sequence[int], x: np.ndarray, rnd) -> List[np.ndarray]:
    """1[A_l > 0] for each hidden layer, with A_l evaluated from operands rounded by `rnd`."""
    ws, bs = unpack(np.asarray(theta, dtype=np.float64), dims)
    h = rnd(x)
    masks = []
    for l in range(len(ws) - 1):
        a = h @ rnd(ws[l]).T + bs[l]
        masks.append(a > 0.0)
        h = rnd(np.maximum(a, 0.0))
    return masks


def cross_entropy_rows(z: np.ndarray, y: np.ndarray):
    """Per-row CE(z_i, y_i) = logsumexp(z_i) - z_{i, y_i} and softmax(z_i)."""
    zmax = z.max(axis=1, keepdims=True)
    e = np.exp(z - zmax)
    s = e.sum(axis=1, keepdims=True)
    lse = zmax[:, 0] + np.log(s[:, 0])
    ce = lse - z[np.arange(z.shape[0]), y]
    return ce, e / s


def worker_loss_grad(theta: np.ndarray, dims: Sequence[int], x_m: np.ndarray,
                     y_m: np.ndarray, decide=None) -> Tuple[float, np.ndarray]:
    """L_m and g^m = grad L_m (flat fp64 [P]) on one worker's segment (Eq. 1).

    decide: None, or an operand rounding (e.g. round_bf16) from which the ReLU' masks are taken."""
    theta = np.asarray(theta, dtype=np.float64)
    ws, _ = unpack(theta, dims)
    lay, p = layout(dims)
    n_m = x_m.shape[0]
    acts, hs = forward(theta, dims, x_m)
    if decide is None:
        masks = [a > 0.0 for a in acts[:-1]]
    else:
        masks = relu_decisions(theta, dims, x_m, decide)
    y_m = np.asarray(y_m, dtype=np.int64)
    ce, prob = cross_entropy_rows(acts[-1], y_m)
    loss = float(ce.sum() / n_m)
    d_a = prob.copy()
    d_a[np.arange(n_m), y_m] -= 1.0
    d_a /= n_m
    g = np.zeros(p, dtype=np.float64)
    for l in range(len(ws) - 1, -1, -1):
        w_off, shape, b_off, o = lay[l]
        g[w_off:w_off + shape[0] * shape[1]] = (d_a.T @ hs[l]).reshape(-1)
        g[b_off:b_off + o] = d_a.sum(axis=0)
        if l > 0:
            d_a = (d_a @ ws[l]) * masks[l - 1]
    return loss, g


def full_batch_loss(theta: np.ndarray, dims: Sequence[int], x: np.ndarray, y: np.ndarray) -> float:
    """Mean CE over all rows (used by the pins: the target of the CP-weighted synchronisation)."""
    acts, _ = forward(theta, dims, x)
    ce, _ = cross_entropy_rows(acts[-1], np.asarray(y, dtype=np.int64))
    return float(ce.mean())
