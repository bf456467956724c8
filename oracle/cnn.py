"""Per-worker loss and gradient of the CNN workload - oracle, fp64 NumPy.

Test infrastructure only (see oracle/__init__.py).

The paper trains ResNet50 / VGG16 on CIFAR10 (Section 5).  The stand-in model
is a small all-conv net on 3x32x32 inputs: three 3x3 convolutions with
padding 1 (strides 1, 2, 2; ReLU after each), global average pooling over the
last feature map, and one fully connected layer to the classes.  The
per-worker objective is again Eq. 1's mean over the worker's samples of
CE(z, y) = logsumexp(z) - z_y.

Convolution is written as its definition, out[n, co, ho, wo] =
b[co] + sum_{ci, kh, kw} x_pad[n, ci, s*ho + kh, s*wo + kw] * W[co, ci, kh, kw],
gathered into explicit patch rows (im2col) so that one matrix product evaluates
the sum; the backward pass is the same sum read the other way (weight gradient
= patches^T dOut, input gradient = scatter-add of dOut W back to the padded
input).  Parameters: flat [conv1.W, conv1.b, conv2.W, conv2.b, conv3.W,
conv3.b, fc.W, fc.b], conv weights [Cout, Cin, 3, 3], fc.W [classes, C3].

`decide` (optional) is the same device as in oracle.mlp: an operand rounding from which
the ReLU' masks are taken (the forward evaluated with rounded input, weights and stored
activations, exact accumulation), so that a bf16 kernel and the oracle take those 0/1
decisions in the same precision; every value stays fp64.
"""
from __future__ import annotations

from typing import Sequence, Tuple

import numpy as np

STRIDES = (1, 2, 2)


def shapes(dims: Sequence[int]):
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


def unpack(theta: np.ndarray, dims: Sequence[int]):
    parts, off = [], 0
    for s in shapes(dims):
        k = int(np.prod(s))
        parts.append(theta[off:off + k].reshape(s))
        off += k
    assert off == theta.size, (off, theta.size)
    return parts


def param_count(dims: Sequence[int]) -> int:
    return int(sum(int(np.prod(s)) for s in shapes(dims)))


def _out_size(h: int, s: int) -> int:
    return (h + 2 - 3) // s + 1


def im2col(h: np.ndarray, s: int) -> np.ndarray:
    """Patch rows [n, Ho, Wo, C, 3, 3] of the zero-padded input."""
    n, c, hh, ww = h.shape
    ho, wo = _out_size(hh, s), _out_size(ww, s)
    hp = np.zeros((n, c, hh + 2, ww + 2), dtype=h.dtype)
    hp[:, :, 1:-1, 1:-1] = h
    col = np.empty((n, ho, wo, c, 3, 3), dtype=h.dtype)
    for kh in range(3):
        for kw in range(3):
            patch = hp[:, :, kh:kh + s * (ho - 1) + 1:s, kw:kw + s * (wo - 1) + 1:s]
            col[:, :, :, :, kh, kw] = patch.transpose(0, 2, 3, 1)
    return col


def col2im(dcol: np.ndarray, in_shape, s: int) -> np.ndarray:
    """Scatter-add of patch-row gradients back onto the input (the adjoint of im2col)."""
    n, c, hh, ww = in_shape
    _, ho, wo = dcol.shape[:3]
    dhp = np.zeros((n, c, hh + 2, ww + 2), dtype=dcol.dtype)
    for kh in range(3):
        for kw in range(3):
            dhp[:, :, kh:kh + s * (ho - 1) + 1:s, kw:kw + s * (wo - 1) + 1:s] += \
                dcol[:, :, :, :, kh, kw].transpose(0, 3, 1, 2)
    return dhp[:, :, 1:-1, 1:-1]


def conv_forward(h: np.ndarray, w: np.ndarray, b: np.ndarray, s: int):
    n = h.shape[0]
    cout = w.shape[0]
    col = im2col(h, s)
    _, ho, wo = col.shape[:3]
    out = col.reshape(n * ho * wo, -1) @ w.reshape(cout, -1).T + b
    return out.reshape(n, ho, wo, cout).transpose(0, 3, 1, 2), col


def forward(theta: np.ndarray, dims: Sequence[int], x: np.ndarray):
    parts = unpack(np.asarray(theta, dtype=np.float64), dims)
    h = np.asarray(x, dtype=np.float64)
    pre, ins, cols = [], [], []
    for k, s in enumerate(STRIDES):
        w, b = parts[2 * k], parts[2 * k + 1]
        ins.append(h)
        a, col = conv_forward(h, w, b, s)
        pre.append(a)
        cols.append(col)
        h = np.maximum(a, 0.0)
    pooled = h.mean(axis=(2, 3))
    z = pooled @ parts[6].T + parts[7]
    return z, dict(pre=pre, ins=ins, cols=cols, last=h, pooled=pooled, parts=parts)


def relu_decisions(theta: np.ndarray, dims: Sequence[int], x: np.ndarray, rnd):
    """1[A_k > 0] for each convolution, with A_k evaluated from operands rounded by `rnd`."""
    parts = unpack(np.asarray(theta, dtype=np.float64), dims)
    h = rnd(x)
    masks = []
    for k, s in enumerate(STRIDES):
        a, _ = conv_forward(h, rnd(parts[2 * k]), parts[2 * k + 1], s)
        masks.append(a > 0.0)
        h = rnd(np.maximum(a, 0.0))
    return masks


def _ce(z: np.ndarray, y: np.ndarray):
    zmax = z.max(axis=1, keepdims=True)
    e = np.exp(z - zmax)
    s = e.sum(axis=1, keepdims=True)
    ce = zmax[:, 0] + np.log(s[:, 0]) - z[np.arange(z.shape[0]), y]
    return ce, e / s


def worker_loss_grad(theta: np.ndarray, dims: Sequence[int], x_m: np.ndarray,
                     y_m: np.ndarray, decide=None) -> Tuple[float, np.ndarray]:
    """L_m and g^m (flat fp64 [P]) on one worker's segment (Eq. 1); decide as in the module doc."""
    theta = np.asarray(theta, dtype=np.float64)
    n_m = x_m.shape[0]
    y_m = np.asarray(y_m, dtype=np.int64)
    z, c = forward(theta, dims, x_m)
    if decide is None:
        masks = [a > 0.0 for a in c["pre"]]
    else:
        masks = relu_decisions(theta, dims, x_m, decide)
    ce, prob = _ce(z, y_m)
    loss = float(ce.sum() / n_m)
    dz = prob.copy()
    dz[np.arange(n_m), y_m] -= 1.0
    dz /= n_m
    parts = c["parts"]
    grads = [None] * 8
    grads[6] = dz.T @ c["pooled"]
    grads[7] = dz.sum(axis=0)
    dpool = dz @ parts[6]
    last = c["last"]
    area = last.shape[2] * last.shape[3]
    dh = np.broadcast_to(dpool[:, :, None, None] / area, last.shape)
    for k in range(len(STRIDES) - 1, -1, -1):
        s = STRIDES[k]
        da = dh * masks[k]
        w = parts[2 * k]
        cout = w.shape[0]
        n, _, ho, wo = da.shape
        da2 = da.transpose(0, 2, 3, 1).reshape(n * ho * wo, cout)
        col2 = c["cols"][k].reshape(n * ho * wo, -1)
        grads[2 * k] = (da2.T @ col2).reshape(w.shape)
        grads[2 * k + 1] = da2.sum(axis=0)
        if k > 0:
            dcol = (da2 @ w.reshape(cout, -1)).reshape(c["cols"][k].shape)
            dh = col2im(dcol, c["ins"][k].shape, s)
    g = np.concatenate([gg.reshape(-1) for gg in grads])
    return loss, g


def full_batch_loss(theta: np.ndarray, dims: Sequence[int], x: np.ndarray, y: np.ndarray) -> float:
    z, _ = forward(theta, dims, x)
    ce, _ = _ce(z, np.asarray(y, dtype=np.int64))
    return float(ce.mean())
