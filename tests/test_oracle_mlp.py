"""Pins for the oracle's MLP gradient, synchronisation and update (Eq. 1, Section 1, Section 4.2).

Independent references: central finite differences in fp64, torch.autograd and
torch.optim.SGD in fp64 on the CPU (library routines, used only here).
"""
import numpy as np
import pytest
import torch

from oracle import mlp, sgd
from oracle import partition as P


def _tiny(dims=(8, 5, 3), n=6, seed=0):
    rng = np.random.default_rng(seed)
    _, p = mlp.layout(dims)
    theta = rng.standard_normal(p) * 0.7
    x = rng.standard_normal((n, dims[0]))
    y = rng.integers(0, dims[-1], n)
    return theta, x, y


def _kink_free(theta, dims, x, margin):
    acts, _ = mlp.forward(theta, dims, x)
    return all(np.abs(a).min() > margin for a in acts[:-1])


def test_finite_differences():
    dims = (8, 5, 4, 3)
    h = 1e-6
    done = 0
    for seed in range(40):
        theta, x, y = _tiny(dims, 5, seed)
        if not _kink_free(theta, dims, x, 10 * h):
            continue
        loss, g = mlp.worker_loss_grad(theta, dims, x, y)
        fd = np.empty_like(theta)
        for j in range(theta.size):
            tp, tm = theta.copy(), theta.copy()
            tp[j] += h
            tm[j] -= h
            fd[j] = (mlp.worker_loss_grad(tp, dims, x, y)[0] - mlp.worker_loss_grad(tm, dims, x, y)[0]) / (2 * h)
        assert np.linalg.norm(fd - g) <= 1e-6 * np.linalg.norm(g), seed
        done += 1
        if done == 3:
            break
    assert done == 3


def _torch_loss(theta, dims, x, y):
    t = torch.tensor(theta, dtype=torch.float64, requires_grad=True)
    h = torch.tensor(x, dtype=torch.float64)
    off = 0
    for l in range(1, len(dims)):
        o, i = dims[l], dims[l - 1]
        w = t[off:off + o * i].view(o, i)
        off += o * i
        b = t[off:off + o]
        off += o
        h = torch.nn.functional.linear(h, w, b)
        if l < len(dims) - 1:
            h = torch.relu(h)
    loss = torch.nn.functional.cross_entropy(h, torch.tensor(y, dtype=torch.long))
    return t, loss


def _torch_grad(theta, dims, x, y):
    t, loss = _torch_loss(theta, dims, x, y)
    loss.backward()
    return loss.item(), t.grad.numpy()


@pytest.mark.parametrize("dims,n", [((8, 5, 3), 7), ((12, 9, 7, 4), 11), ((3072, 64, 10), 32)])
def test_matches_torch_autograd(dims, n):
    theta, x, y = _tiny(dims, n, 3)
    lo, go = mlp.worker_loss_grad(theta, dims, x, y)
    lt, gt = _torch_grad(theta, dims, x, y)
    assert abs(lo - lt) <= 1e-12 * abs(lt)
    assert np.linalg.norm(go - gt) <= 1e-11 * np.linalg.norm(gt)


def test_cp_weighted_sync_is_full_batch_gradient():
    # Mean per-worker losses (Eq. 1) weighted by n_m / N sum to the full-batch mean loss.
    dims = (10, 7, 5)
    theta, x, y = _tiny(dims, 37, 4)
    _, g_full = _torch_grad(theta, dims, x, y)
    for cp in ([1, 3], [1, 1, 2, 4], [5, 1, 1, 1, 3], [1.0]):
        sizes = P.partition_sizes(cp, 37)
        _, loss, g, _, _ = sgd.step(mlp.worker_loss_grad, theta, dims, x, y, sizes, 0.0, sgd.SYNC_CP_WEIGHTED)
        assert np.linalg.norm(g - g_full) <= 1e-12 * np.linalg.norm(g_full)
        assert abs(loss - mlp.full_batch_loss(theta, dims, x, y)) < 1e-12


def test_mean_sync_closed_form():
    # Section 1: g = (1/M) sum_m g^m, each g^m the gradient of worker m's mean loss.
    dims = (10, 7, 5)
    theta, x, y = _tiny(dims, 40, 5)
    sizes = P.partition_sizes([1, 2, 3, 6], 40)
    off = P.offsets(sizes)
    want = sum(_torch_grad(theta, dims, x[off[m]:off[m + 1]], y[off[m]:off[m + 1]])[1]
               for m in range(4)) / 4
    _, _, g, slabs, losses = sgd.step(mlp.worker_loss_grad, theta, dims, x, y, sizes, 0.0, sgd.SYNC_MEAN,
                                      keep_slabs=True)
    assert np.linalg.norm(g - want) <= 1e-12 * np.linalg.norm(want)
    # unequal partitions: the plain average is not the full-batch gradient
    _, g_full = _torch_grad(theta, dims, x, y)
    assert np.linalg.norm(g - g_full) > 1e-3 * np.linalg.norm(g_full)
    # equal partitions: it is
    sizes_eq = P.even_sizes(4, 40)
    _, _, g_eq, _, _ = sgd.step(mlp.worker_loss_grad, theta, dims, x, y, sizes_eq, 0.0, sgd.SYNC_MEAN)
    assert np.linalg.norm(g_eq - g_full) <= 1e-12 * np.linalg.norm(g_full)


def test_update_matches_torch_sgd():
    # theta_{t+1} = theta_t - eta g_t, three steps, against torch.optim.SGD on the full-batch loss.
    dims = (9, 6, 4)
    theta, x, y = _tiny(dims, 24, 6)
    sizes = P.partition_sizes([1, 2, 5], 24)
    lr = 0.3
    t = torch.tensor(theta, dtype=torch.float64, requires_grad=True)
    opt = torch.optim.SGD([t], lr=lr)
    th = theta.copy()
    for _ in range(3):
        opt.zero_grad()
        _, loss = _torch_loss(t.detach().numpy(), dims, x, y)
        # rebuild the graph on t itself
        h = torch.tensor(x, dtype=torch.float64)
        off = 0
        for l in range(1, len(dims)):
            o, i = dims[l], dims[l - 1]
            w = t[off:off + o * i].view(o, i)
            off += o * i
            b = t[off:off + o]
            off += o
            h = torch.nn.functional.linear(h, w, b)
            if l < len(dims) - 1:
                h = torch.relu(h)
        torch.nn.functional.cross_entropy(h, torch.tensor(y, dtype=torch.long)).backward()
        opt.step()
        th, _, _, _, _ = sgd.step(mlp.worker_loss_grad, th, dims, x, y, sizes, lr, sgd.SYNC_CP_WEIGHTED)
    assert np.allclose(th, t.detach().numpy(), rtol=0, atol=1e-12)


def test_single_worker_is_plain_sgd():
    dims = (6, 4, 3)
    theta, x, y = _tiny(dims, 9, 7)
    for mode in (sgd.SYNC_MEAN, sgd.SYNC_CP_WEIGHTED):
        th1, loss, g, _, _ = sgd.step(mlp.worker_loss_grad, theta, dims, x, y, [9], 0.1, mode)
        lt, gt = _torch_grad(theta, dims, x, y)
        assert np.allclose(th1, theta - 0.1 * gt, atol=1e-13)
        assert abs(loss - lt) < 1e-12


def test_sync_weights():
    assert np.allclose(sgd.sync_weights([32, 96], sgd.SYNC_MEAN), [0.5, 0.5])
    assert np.allclose(sgd.sync_weights([32, 96], sgd.SYNC_CP_WEIGHTED), [0.25, 0.75])
    w = sgd.sync_weights([43, 85, 128, 256], sgd.SYNC_CP_LITERAL, cp=[1, 2, 3, 6])
    assert np.allclose(w, np.array([1, 2, 3, 6]) / 12 / 4)


def test_loss_decreases():
    dims = (16, 12, 4)
    theta, x, y = _tiny(dims, 64, 8)
    theta *= 0.5
    sizes = P.partition_sizes([1, 3], 64)
    losses = []
    for _ in range(5):
        theta, loss, _, _, _ = sgd.step(mlp.worker_loss_grad, theta, dims, x, y, sizes, 0.05, sgd.SYNC_CP_WEIGHTED)
        losses.append(loss)
    assert all(b < a for a, b in zip(losses, losses[1:]))


def test_round_bf16_matches_torch():
    rng = np.random.default_rng(0)
    vals = np.concatenate([
        rng.standard_normal(20000).astype(np.float32) * np.float32(10.0) ** rng.integers(-30, 30, 20000),
        rng.standard_normal(1000).astype(np.float32) * np.float32(1e-39),      # fp32 subnormals
    ]).astype(np.float32)
    # exact ties: low 16 bits = 0x8000, with even and odd kept parts
    base = rng.integers(0x3F800000, 0x40800000, 2000, dtype=np.uint32) & np.uint32(0xFFFF0000)
    ties = (base | np.uint32(0x8000)).view(np.float32)
    vals = np.concatenate([vals, ties, -ties, np.array([0.0, -0.0, 1.0, -1.0], dtype=np.float32)])
    want = torch.from_numpy(vals).to(torch.bfloat16).to(torch.float64).numpy()
    got = mlp.round_bf16(vals)
    assert np.array_equal(got, want)


def test_decision_mode_identity_rounding_is_exact_oracle():
    dims = (12, 9, 7, 4)
    theta, x, y = _tiny(dims, 11, 3)
    l0, g0 = mlp.worker_loss_grad(theta, dims, x, y)
    l1, g1 = mlp.worker_loss_grad(theta, dims, x, y, decide=lambda a: np.asarray(a, dtype=np.float64))
    assert l0 == l1 and np.array_equal(g0, g1)


def test_bf16_decisions_differ_only_near_kinks():
    # A decision taken from bf16-rounded operands can only disagree with the exact one where the
    # exact pre-activation lies within the bf16 rounding of the operands (|A| small).
    dims = (256, 128, 64, 10)
    rng = np.random.default_rng(4)
    _, p = mlp.layout(dims)
    theta = rng.standard_normal(p) * 0.1
    x = rng.standard_normal((200, 256))
    acts, _ = mlp.forward(theta, dims, x)
    masks = mlp.relu_decisions(theta, dims, x, mlp.round_bf16)
    flips = 0
    for a, m in zip(acts[:-1], masks):
        diff = (a > 0) != m
        flips += int(diff.sum())
        if diff.any():
            assert np.abs(a[diff]).max() < 0.05 * np.abs(a).std()
    assert flips < 0.01 * sum(a.size for a in acts[:-1])
    # and the gradient with bf16 decisions stays close to the exact one
    _, g0 = mlp.worker_loss_grad(theta, dims, x[:50], y := rng.integers(0, 10, 50))
    _, g1 = mlp.worker_loss_grad(theta, dims, x[:50], y, decide=mlp.round_bf16)
    assert np.linalg.norm(g1 - g0) < 0.2 * np.linalg.norm(g0)


def test_momentum_weight_decay_matches_torch_sgd():
    # Section 5: SGD with momentum 0.9 and weight decay 5e-4, against torch.optim.SGD in fp64.
    dims = (9, 6, 4)
    theta, x, y = _tiny(dims, 24, 11)
    sizes = P.partition_sizes([1, 2, 5], 24)
    lr, mu, wd = 0.2, 0.9, 5e-4
    t = torch.tensor(theta, dtype=torch.float64, requires_grad=True)
    opt = torch.optim.SGD([t], lr=lr, momentum=mu, weight_decay=wd)
    th, buf = theta.copy(), None
    for _ in range(5):
        opt.zero_grad()
        tt, loss = _torch_loss(t.detach().numpy(), dims, x, y)
        loss.backward()
        t.grad = tt.grad.clone()
        opt.step()
        _, _, g, _, _ = sgd.step(mlp.worker_loss_grad, th, dims, x, y, sizes, 0.0, sgd.SYNC_CP_WEIGHTED)
        th, buf = sgd.momentum_update(th, g, buf, lr, mu, wd)
    assert np.allclose(th, t.detach().numpy(), rtol=0, atol=1e-12)


def test_cosine_lr_matches_torch_scheduler():
    p = torch.nn.Parameter(torch.zeros(1))
    opt = torch.optim.SGD([p], lr=0.1)
    sched = torch.optim.lr_scheduler.CosineAnnealingLR(opt, T_max=50, eta_min=0.001)
    for step in range(50):
        assert abs(opt.param_groups[0]["lr"] - sgd.cosine_lr(0.1, 0.001, step, 50)) < 1e-12
        opt.step()
        sched.step()
