"""Pins for the oracle's CNN gradient: finite differences and torch.autograd (fp64, CPU)."""
import numpy as np
import torch

import synth
from oracle import cnn, sgd
from oracle import partition as P

TINY = (2, 6, 6, 3, 4, 5, 3)        # Cin, H, W, c1, c2, c3, classes


def _tiny(dims=TINY, n=3, seed=0):
    rng = np.random.default_rng(seed)
    theta = rng.standard_normal(cnn.param_count(dims)) * 0.6
    x = rng.standard_normal((n,) + tuple(dims[:3]))
    y = rng.integers(0, dims[-1], n)
    return theta, x, y


def _torch_grad(theta, dims, x, y):
    t = torch.tensor(theta, dtype=torch.float64, requires_grad=True)
    parts, off = [], 0
    for s in cnn.shapes(dims):
        k = int(np.prod(s))
        parts.append(t[off:off + k].view(s))
        off += k
    h = torch.tensor(x, dtype=torch.float64)
    for k, s in enumerate(cnn.STRIDES):
        h = torch.relu(torch.nn.functional.conv2d(h, parts[2 * k], parts[2 * k + 1], stride=s, padding=1))
    z = torch.nn.functional.linear(h.mean(dim=(2, 3)), parts[6], parts[7])
    loss = torch.nn.functional.cross_entropy(z, torch.tensor(y, dtype=torch.long))
    loss.backward()
    return loss.item(), t.grad.numpy()


def test_param_count_matches_layout():
    assert cnn.param_count(synth.WORKLOADS[synth.CFG4].dims) == 373386
    assert synth.param_count(synth.CNN, synth.WORKLOADS[synth.CFG4].dims) == 373386


def test_im2col_adjoint():
    # <im2col(x), c> == <x, col2im(c)> for random x, c: col2im is the adjoint of the gather.
    rng = np.random.default_rng(2)
    for s in (1, 2):
        x = rng.standard_normal((2, 3, 7, 6))
        col = cnn.im2col(x, s)
        c = rng.standard_normal(col.shape)
        assert abs(np.sum(col * c) - np.sum(x * cnn.col2im(c, x.shape, s))) < 1e-10


def test_finite_differences():
    h = 1e-6
    done = 0
    for seed in range(60):
        theta, x, y = _tiny(seed=seed)
        _, c = cnn.forward(theta, TINY, x)
        if min(np.abs(a).min() for a in c["pre"]) < 10 * h:
            continue
        loss, g = cnn.worker_loss_grad(theta, TINY, x, y)
        fd = np.empty_like(theta)
        for j in range(theta.size):
            tp, tm = theta.copy(), theta.copy()
            tp[j] += h
            tm[j] -= h
            fd[j] = (cnn.worker_loss_grad(tp, TINY, x, y)[0] - cnn.worker_loss_grad(tm, TINY, x, y)[0]) / (2 * h)
        assert np.linalg.norm(fd - g) <= 1e-6 * np.linalg.norm(g), seed
        done += 1
        if done == 2:
            break
    assert done == 2


def test_matches_torch_autograd():
    for dims, n in ((TINY, 4), ((3, 32, 32, 8, 12, 16, 10), 5)):
        theta, x, y = _tiny(dims, n, 9)
        lo, go = cnn.worker_loss_grad(theta, dims, x, y)
        lt, gt = _torch_grad(theta, dims, x, y)
        assert abs(lo - lt) <= 1e-12 * abs(lt)
        assert np.linalg.norm(go - gt) <= 1e-11 * np.linalg.norm(gt)


def test_cp_weighted_is_full_batch():
    theta, x, y = _tiny(TINY, 12, 3)
    _, g_full = _torch_grad(theta, TINY, x, y)
    sizes = P.partition_sizes([1, 2, 3, 6], 12)
    _, _, g, _, _ = sgd.step(cnn.worker_loss_grad, theta, TINY, x, y, sizes, 0.0, sgd.SYNC_CP_WEIGHTED)
    assert np.linalg.norm(g - g_full) <= 1e-12 * np.linalg.norm(g_full)


def test_decision_mode_identity_is_exact():
    theta, x, y = _tiny(TINY, 4, 5)
    l0, g0 = cnn.worker_loss_grad(theta, TINY, x, y)
    l1, g1 = cnn.worker_loss_grad(theta, TINY, x, y, decide=lambda a: np.asarray(a, dtype=np.float64))
    assert l0 == l1 and np.array_equal(g0, g1)


def test_bf16_decisions_differ_only_near_kinks():
    from oracle import mlp
    dims = (3, 16, 16, 16, 24, 32, 10)
    theta, x, y = _tiny(dims, 6, 8)
    theta *= 0.5
    _, c = cnn.forward(theta, dims, x)
    masks = cnn.relu_decisions(theta, dims, x, mlp.round_bf16)
    flips = 0
    for a, m in zip(c["pre"], masks):
        diff = (a > 0) != m
        flips += int(diff.sum())
        if diff.any():
            assert np.abs(a[diff]).max() < 0.05 * np.abs(a).std()
    assert flips < 0.01 * sum(a.size for a in c["pre"])
