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


# ---------------------------------------------------------------------------------------------
# Hand-worked pins of the ReLU'-decision mode on a 1x1 image with one channel per layer.  With
# padding 1 a 3x3 convolution of a 1x1 image reads the real pixel through its centre tap only; the
# eight other taps multiply the zero padding (set to 5 here, so any padding mistake shows), and
# every stride gives a 1x1 output.  The net is then a chain of scalars: A_k = c_k h_{k-1} + b_k,
# h_k = ReLU(A_k), pooled = h_3, z = [h_3, -h_3] (fc W = [[1], [-1]], b = 0), y = 0, so
# dL/dh_3 = -2 sigmoid(-2 h_3), dL/dA_k = dL/dh_k * mask_k, dL/dh_{k-1} = c_k dL/dA_k.
# bf16 keeps 8 significant bits: 1 + 2^-8 is a tie that rounds to 1, 1 - 2^-10 rounds to 1.
E8, E9, E10 = 2.0 ** -8, 2.0 ** -9, 2.0 ** -10
ONE = (1, 1, 1, 1, 1, 1, 2)


def _chain(x, centres, biases):
    parts = []
    for c, b in zip(centres, biases):
        w = np.full((3, 3), 5.0)
        w[1, 1] = c
        parts += list(w.ravel()) + [b]
    parts += [1.0, -1.0, 0.0, 0.0]
    return np.asarray(parts, dtype=np.float64), np.array([[[[x]]]])


def _hand_grad(x, centres, biases, masks):
    """The gradient of the scalar chain written out: values exact, decisions as given."""
    h = [x]
    for c, b in zip(centres, biases):
        h.append(max(c * h[-1] + b, 0.0))
    s = 1.0 / (1.0 + np.exp(2.0 * h[3]))                 # sigmoid(-2 h3)
    p0 = 1.0 - s
    dh = -2.0 * s
    g = [None] * 3
    for k in (2, 1, 0):
        da = dh * masks[k]
        gw = np.zeros(9)
        gw[4] = da * h[k]
        g[k] = list(gw) + [da]
        dh = da * centres[k]
    return np.asarray(g[0] + g[1] + g[2] + [(p0 - 1.0) * h[3], (1.0 - p0) * h[3], p0 - 1.0, 1.0 - p0])


def _cnn_masks(theta, x, rnd):
    return [bool(m.ravel()[0]) for m in cnn.relu_decisions(theta, ONE, x, rnd)]


def _exact(a):
    return np.asarray(a, dtype=np.float64)


def _check_case(x, centres, biases, want):
    """want: {rounding: masks}; the gradient with each rounding's decisions equals the chain's."""
    from oracle import mlp
    theta, xa = _chain(x, centres, biases)
    for name, masks in want.items():
        rnd = {"bf16": mlp.round_bf16, "fp32": mlp.round_fp32, "exact": _exact}[name]
        assert _cnn_masks(theta, xa, rnd) == masks, name
        kw = {} if name == "exact" else {"decide": rnd}
        _, g = cnn.worker_loss_grad(theta, ONE, xa, np.array([0]), **kw)
        assert np.allclose(g, _hand_grad(x, centres, biases, masks), rtol=1e-14, atol=1e-300), name
        assert np.all(g[[k for k in range(30) if k % 10 not in (4, 9)]] == 0.0)   # padding taps


def test_hand_pin_input_rounding_flips_first_conv():
    # x = 1 + 2^-8, c1 = 1, b1 = -(1 + 2^-9): exact A1 = 2^-9 > 0, bf16 A1 = 1 - (1 + 2^-9) < 0.
    # b2 = 1 keeps conv 2 (and conv 3) on whatever h1 is.
    _check_case(1.0 + E8, [1.0, 1.0, 1.0], [-(1.0 + E9), 1.0, 0.0],
                {"bf16": [False, True, True], "fp32": [True, True, True], "exact": [True, True, True]})


def test_hand_pin_weight_rounding_flips_first_conv():
    _check_case(1.0, [1.0 + E8, 1.0, 1.0], [-(1.0 + E9), 1.0, 0.0],
                {"bf16": [False, True, True], "fp32": [True, True, True]})


def test_hand_pin_conv_bias_is_not_rounded():
    # b1 = -(1 - 2^-10) as stored gives A1 = 2^-10 > 0; a bf16-rounded bias (-1) would give 0 (off).
    _check_case(1.0, [1.0, 1.0, 1.0], [-(1.0 - E10), 1.0, 0.0], {"bf16": [True, True, True]})


def test_hand_pin_stored_activation_rounding_flips_second_conv():
    # A1 = 1 + 2^-8 in every precision; the stored h1 rounds to 1 in bf16, so with c2 = 1,
    # b2 = -(1 + 2^-9) the exact A2 = 2^-9 is on and the bf16 A2 = -2^-9 is off.  b3 = 1 keeps conv 3
    # on, so the flip shows in the gradient: nothing reaches conv 2 or conv 1 under bf16 decisions.
    _check_case(1.0, [1.0, 1.0, 1.0], [E8, -(1.0 + E9), 1.0],
                {"bf16": [True, False, True], "fp32": [True, True, True], "exact": [True, True, True]})


def test_hand_pin_fp32_rounding_of_stored_conv_activations():
    # x = 1, c1 = 1, b1 = 2^-30: A1 = 1 + 2^-30, stored in fp32 as 1; c2 = 1, b2 = -1: exact A2 = 2^-30
    # (on), fp32 A2 = 0 (off, ReLU'(0) = 0).
    _check_case(1.0, [1.0, 1.0, 1.0], [2.0 ** -30, -1.0, 1.0],
                {"fp32": [True, False, True], "exact": [True, True, True]})
