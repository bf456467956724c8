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


# ---------------------------------------------------------------------------------------------
# Hand-worked pins of the ReLU'-decision mode.  Each net has one hidden unit per layer, one
# sample and two classes with W_out = [[1], [-1]], b_out = 0, y = 0, so the arithmetic fits in a
# comment.  The operands sit next to bf16 ties: bf16 keeps 8 significant bits, so between 1 and 2
# the representable values are 2^-7 apart, 1 + 2^-8 is a tie (rounds to the even 1), and
# 1 - 2^-10 rounds to 1.  With last hidden activation h the logits are z = [h, -h], softmax
# p0 = sigmoid(2h), and dL/dh = (p0 - 1) - (1 - p0) = -2 sigmoid(-2h).
E8, E9, E10 = 2.0 ** -8, 2.0 ** -9, 2.0 ** -10


def _sigmoid(v):
    return 1.0 / (1.0 + np.exp(-v))


def _one_unit_net(ws, bs):
    """Flat theta of an MLP with one unit per hidden layer and the fixed two-class output layer."""
    parts = []
    for w, b in zip(ws, bs):
        parts += list(np.ravel(w)) + [b]
    parts += [1.0, -1.0, 0.0, 0.0]
    return np.asarray(parts, dtype=np.float64)


def _masks(theta, dims, x, rnd):
    return [bool(m[0, 0]) for m in mlp.relu_decisions(theta, dims, x, rnd)]


def test_hand_pin_input_rounding_flips_first_layer():
    # x = 1 + 2^-8, W1 = 1, b1 = -(1 + 2^-9): exact A1 = 2^-9 > 0.  bf16(x) = 1 (tie to even), so
    # the bf16 decision sees 1 - (1 + 2^-9) = -2^-9 < 0.  x is an fp32 value: fp32 keeps the unit.
    dims = (1, 1, 2)
    x = np.array([[1.0 + E8]])
    theta = _one_unit_net([[1.0]], [-(1.0 + E9)])
    assert _masks(theta, dims, x, mlp.round_bf16) == [False]
    assert _masks(theta, dims, x, mlp.round_fp32) == [True]
    h = E9
    d = -2.0 * _sigmoid(-2.0 * h)                       # dL/dA1 when the unit is on
    loss, g_exact = mlp.worker_loss_grad(theta, dims, x, [0])
    _, g_bf16 = mlp.worker_loss_grad(theta, dims, x, [0], decide=mlp.round_bf16)
    assert abs(loss - np.log1p(np.exp(-2.0 * h))) <= 1e-15
    # layout [W1, b1, W2 (2x1), b2 (2)]
    p0 = _sigmoid(2.0 * h)
    want_exact = [d * (1.0 + E8), d, (p0 - 1.0) * h, (1.0 - p0) * h, p0 - 1.0, 1.0 - p0]
    want_bf16 = [0.0, 0.0] + want_exact[2:]              # unit off: no signal reaches W1, b1
    assert np.allclose(g_exact, want_exact, rtol=1e-14, atol=0)
    assert np.allclose(g_bf16, want_bf16, rtol=1e-14, atol=0)
    assert g_bf16[0] == 0.0 and g_bf16[1] == 0.0


def test_hand_pin_weight_rounding_flips_first_layer():
    # The same with the off-grid value in the weight: x = 1, W1 = 1 + 2^-8.
    dims = (1, 1, 2)
    x = np.array([[1.0]])
    theta = _one_unit_net([[1.0 + E8]], [-(1.0 + E9)])
    assert _masks(theta, dims, x, mlp.round_bf16) == [False]
    assert _masks(theta, dims, x, mlp.round_fp32) == [True]
    _, g = mlp.worker_loss_grad(theta, dims, x, [0], decide=mlp.round_bf16)
    assert g[0] == 0.0 and g[1] == 0.0
    _, g = mlp.worker_loss_grad(theta, dims, x, [0])
    assert np.isclose(g[0], -2.0 * _sigmoid(-2.0 * E9), rtol=1e-14, atol=0)


def test_hand_pin_bias_is_not_rounded():
    # The kernels add the fp32 bias to the fp32 accumulator: only products see bf16 operands.
    # x = 1, W1 = 1, b1 = -(1 - 2^-10): A1 = 2^-10 > 0 with the bias as stored; a bf16-rounded
    # bias (-1) would give A1 = 0 and switch the unit off (ReLU'(0) = 0).
    dims = (1, 1, 2)
    x = np.array([[1.0]])
    theta = _one_unit_net([[1.0]], [-(1.0 - E10)])
    assert mlp.round_bf16(np.array([-(1.0 - E10)]))[0] == -1.0     # the premise
    assert _masks(theta, dims, x, mlp.round_bf16) == [True]
    _, g = mlp.worker_loss_grad(theta, dims, x, [0], decide=mlp.round_bf16)
    d = -2.0 * _sigmoid(-2.0 * E10)
    assert np.allclose(g[:2], [d, d], rtol=1e-14, atol=0)


def test_hand_pin_rounding_can_switch_a_unit_on():
    # x = 1 + 2^-7 - 2^-9 rounds up to 1 + 2^-7 (0.75 of a bf16 step); b1 = -(1 + 2^-7 - 2^-10):
    # exact A1 = -2^-10 (off), bf16 A1 = +2^-10 (on).  The values stay fp64: h = ReLU(exact A1) = 0,
    # z = [0, 0], p0 = 1/2, so dL/dA1 = 2 (1/2 - 1) = -1 reaches W1 and b1 through the bf16 mask.
    dims = (1, 1, 2)
    xv = 1.0 + 2.0 ** -7 - E9
    x = np.array([[xv]])
    theta = _one_unit_net([[1.0]], [-(1.0 + 2.0 ** -7 - E10)])
    assert _masks(theta, dims, x, mlp.round_bf16) == [True]
    assert _masks(theta, dims, x, mlp.round_fp32) == [False]
    _, g = mlp.worker_loss_grad(theta, dims, x, [0], decide=mlp.round_bf16)
    assert np.allclose(g, [-xv, -1.0, 0.0, 0.0, -0.5, 0.5], rtol=1e-15, atol=0)
    _, g = mlp.worker_loss_grad(theta, dims, x, [0])
    assert np.allclose(g, [0.0, 0.0, 0.0, 0.0, -0.5, 0.5], rtol=1e-15, atol=0)


def test_hand_pin_stored_activation_rounding_flips_second_layer():
    # x = 1, W1 = 1, b1 = 2^-8: A1 = 1 + 2^-8 in every precision (x and W1 are bf16 values, the bias
    # is not rounded), so layer 1 is on everywhere.  The stored activation H1 = 1 + 2^-8 rounds to 1
    # in bf16; with W2 = 1, b2 = -(1 + 2^-9) the exact A2 = 2^-9 > 0 but the bf16 A2 = -2^-9.  Only the
    # rounding of H1 flips layer 2.
    dims = (1, 1, 1, 2)
    x = np.array([[1.0]])
    theta = _one_unit_net([[1.0], [1.0]], [E8, -(1.0 + E9)])
    assert _masks(theta, dims, x, mlp.round_bf16) == [True, False]
    assert _masks(theta, dims, x, mlp.round_fp32) == [True, True]
    h2 = E9
    d = -2.0 * _sigmoid(-2.0 * h2)
    p0 = _sigmoid(2.0 * h2)
    out = [(p0 - 1.0) * h2, (1.0 - p0) * h2, p0 - 1.0, 1.0 - p0]
    # layout [W1, b1, W2, b2, W3 (2x1), b3 (2)]; dL/dA2 = d, dL/dA1 = d * W2 = d, H1 = 1 + 2^-8
    _, g = mlp.worker_loss_grad(theta, dims, x, [0])
    assert np.allclose(g, [d * 1.0, d, d * (1.0 + E8), d] + out, rtol=1e-14, atol=0)
    _, g = mlp.worker_loss_grad(theta, dims, x, [0], decide=mlp.round_bf16)
    assert np.allclose(g, [0.0, 0.0, 0.0, 0.0] + out, rtol=1e-14, atol=0)


def test_hand_pin_fp32_rounding_of_stored_activations():
    # The fp32 check path stores fp32 activations.  x = [1, 2^-30], W1 = [1, 1], b1 = 0: A1 = 1 + 2^-30
    # in fp64, which fp32 (24 significant bits) rounds to 1.  W2 = 1, b2 = -1: exact A2 = 2^-30 > 0, fp32
    # A2 = 0, off (ReLU'(0) = 0).  bf16 agrees with fp32 here; the exact oracle keeps the unit.
    dims = (2, 1, 1, 2)
    x = np.array([[1.0, 2.0 ** -30]])
    theta = _one_unit_net([[1.0, 1.0], [1.0]], [0.0, -1.0])
    assert _masks(theta, dims, x, mlp.round_fp32) == [True, False]
    assert _masks(theta, dims, x, mlp.round_bf16) == [True, False]
    assert _masks(theta, dims, x, lambda a: np.asarray(a, dtype=np.float64)) == [True, True]
    _, g = mlp.worker_loss_grad(theta, dims, x, [0], decide=mlp.round_fp32)
    assert np.all(g[:4] == 0.0)
    _, g = mlp.worker_loss_grad(theta, dims, x, [0])
    d = -2.0 * _sigmoid(-2.0 * 2.0 ** -30)
    assert np.allclose(g[:5], [d, d * 2.0 ** -30, d, d * (1.0 + 2.0 ** -30), d], rtol=1e-14, atol=0)
