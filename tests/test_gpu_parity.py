"""GPU step vs the fp64 oracle on identical seeded inputs.

Acceptance: partitions and index maps bit-exact; the first step's synchronised gradient within
relative L2 1e-2 (bf16 path) or 1e-5 (fp32 check path); parameters after 10 steps within relative
L2 2e-2, also checked on the parameter change theta_10 - theta_0 (a stricter reading: 5e-2 for
bf16, whose rounding biases the small last-layer bias updates - the CPU emulation of the bf16
arithmetic in tests/bf16_emulation.py gives 2.9e-2 on 3072-1024-1024-10 at lr 0.05 - and 2e-3 for
fp32, where one ReLU kink decided differently by fp32 accumulation moves the trajectory by ~1e-3).
For the bf16 path the oracle takes the ReLU' decisions in the kernel's precision (bf16 operands);
every value it computes stays fp64 (a departure from taking them exactly, bounded separately in
test_bf16_against_exact_decisions)."""
import functools
import types

import numpy as np
import pytest
import torch

import synth
import paper_2110_08941_gb300 as hs
from oracle import partition as P
from oracle import mlp
from tests.bf16_emulation import BOUND_DTHETA, BOUND_LOSS_AFTER_FIRST, BOUND_VS_EXACT_DECISIONS
from tests.gpu_helpers import decide_for, rel, run_library, run_oracle

pytestmark = pytest.mark.gpu

TOL_G = {hs.HS_BF16: 1e-2, hs.HS_FP32_CHECK: 1e-5}
TOL_THETA = 2e-2


def _check(lib, orc, theta0, precision, n_steps):
    assert lib["counts"] == orc["counts"]
    for counts, im in zip(lib["counts"], lib["index_maps"]):
        assert np.array_equal(im, np.asarray(P.index_map(counts), dtype=np.int32))
    assert rel(lib["g_first"], orc["g_first"]) <= TOL_G[precision]
    assert rel(lib["theta"], orc["theta"]) <= TOL_THETA
    d_lib, d_orc = lib["theta"] - theta0, orc["theta"] - theta0
    assert rel(d_lib, d_orc) <= (BOUND_DTHETA if precision == hs.HS_BF16 else 2e-3)
    ltol = 1e-2 if precision == hs.HS_BF16 else 1e-5
    # the first loss is at identical parameters; later ones follow the bf16 trajectory, whose loss
    # drifts by up to 1.2e-2 from the oracle's on 3072-1024-1024-10 at lr 0.05 in the CPU emulation
    # of the bf16 arithmetic
    for t, (a, b) in enumerate(zip(lib["losses"], orc["losses"])):
        tol = ltol if (t == 0 or precision != hs.HS_BF16) else BOUND_LOSS_AFTER_FIRST
        assert abs(a - b) <= tol * abs(b), t
    for a, b in zip(lib["worker_losses_first"], orc["worker_losses_first"]):
        assert abs(a - b) <= ltol * abs(b)


CASES = [
    # name, precision, sync
    (synth.CFG1, hs.HS_FP32_CHECK, hs.HS_SYNC_CP_WEIGHTED),
    (synth.CFG1, hs.HS_FP32_CHECK, hs.HS_SYNC_MEAN),
    (synth.CFG1, hs.HS_BF16, hs.HS_SYNC_CP_WEIGHTED),
    (synth.CFG1, hs.HS_BF16, hs.HS_SYNC_MEAN),
    (synth.CFG1, hs.HS_BF16, hs.HS_SYNC_CP_LITERAL),
    (synth.CFG2, hs.HS_FP32_CHECK, hs.HS_SYNC_CP_WEIGHTED),
    (synth.CFG2, hs.HS_BF16, hs.HS_SYNC_CP_WEIGHTED),
    (synth.CFG2, hs.HS_BF16, hs.HS_SYNC_MEAN),
]


@functools.lru_cache(maxsize=None)
def _inputs(name):
    wl = synth.WORKLOADS[name]
    x, y = synth.make_batch(wl)
    return wl, x, y, synth.make_params(wl), synth.initial_weights(wl)


@functools.lru_cache(maxsize=None)
def _oracle_run(name, sync, steps, precision):
    wl, x, y, theta0, w = _inputs(name)
    return run_oracle(wl.arch, wl.dims, wl.workers, wl.global_batch, w, x, y, theta0, wl.lr, steps, sync,
                      decide=decide_for(precision))


@pytest.mark.parametrize("name,precision,sync", CASES)
def test_workload_10_steps(name, precision, sync):
    wl, x, y, theta0, w = _inputs(name)
    steps = 10
    lib = run_library(wl.arch, wl.dims, wl.workers, wl.global_batch, w, x, y, theta0, wl.lr, steps, precision, sync)
    orc = _oracle_run(name, sync, steps, precision)
    _check(lib, orc, theta0.astype(np.float64), precision, steps)


def test_drift_workload_repartition():
    """3072->2048->2048->10, N=4096, M=8, seeded drifting worker speeds: the partition is recomputed
    from windowed throughputs (Eq. 2) between steps; two steps keep the oracle inside the test budget."""
    wl = synth.WORKLOADS[synth.CFG3]
    x, y = synth.make_batch(wl)
    theta0 = synth.make_params(wl)
    speeds = synth.drift_walk(wl.workers, 20, wl.seed)
    rep = {1: list(synth.window_throughputs(speeds[0:10]))}
    lib = run_library(wl.arch, wl.dims, wl.workers, wl.global_batch, None, x, y, theta0, wl.lr, 2, hs.HS_BF16,
                      hs.HS_SYNC_CP_WEIGHTED, repartition=rep)
    orc = run_oracle(wl.arch, wl.dims, wl.workers, wl.global_batch, None, x, y, theta0, wl.lr, 2,
                     hs.HS_SYNC_CP_WEIGHTED, repartition=rep, decide=mlp.round_bf16)
    assert lib["counts"][0] == [512] * 8 and lib["counts"][1] != lib["counts"][0]
    _check(lib, orc, theta0.astype(np.float64), hs.HS_BF16, 2)


@pytest.mark.parametrize("precision", [hs.HS_BF16, hs.HS_FP32_CHECK])
def test_cnn_repartition(precision):
    """The CNN with a repartition between steps (Algorithm 1 on new throughputs): the split-K
    weight-gradient plans, chunk tables and index map are rebuilt for the new segments."""
    dims, N, M = (3, 16, 16, 64, 128, 64, 7), 24, 3
    rng = np.random.default_rng(11)
    x = rng.standard_normal((N,) + tuple(dims[:3]), dtype=np.float32)
    y = rng.integers(0, dims[-1], N, dtype=np.int32)
    theta0 = synth.he_normal_params(synth.CNN, dims, 3)
    rep = {2: [1.0, 4.0, 2.0]}
    lib = run_library(synth.CNN, dims, M, N, [3.0, 1.0, 1.0], x, y, theta0, 0.05, 4, precision,
                      hs.HS_SYNC_CP_WEIGHTED, repartition=rep)
    orc = run_oracle(synth.CNN, dims, M, N, [3.0, 1.0, 1.0], x, y, theta0, 0.05, 4, hs.HS_SYNC_CP_WEIGHTED,
                     repartition=rep, decide=decide_for(precision))
    assert lib["counts"] == [[14, 5, 5], [3, 14, 7]]
    _check(lib, orc, theta0.astype(np.float64), precision, 4)


EDGE = [
    # dims, N, M, weights: one sample per worker; ragged tails in every GEMM dimension; M = 1
    ((24, 16, 3), 5, 5, None),
    ((64, 40, 7), 300, 3, [1.0, 1.0, 5.0]),
    ((136, 264, 136, 1000), 517, 7, [0.3, 2.0, 1.0, 1.0, 0.7, 4.0, 0.01]),
    ((32, 8), 130, 1, None),
    ((40, 48, 56, 9), 257, 40, None),
    # 16 classes (the widest output whose softmax, loss and bias gradient run in one launch), a
    # worker of more than 512 rows; 23 classes (the loss reduction with the bias gradient)
    ((40, 24, 16), 1100, 2, [1.0, 3.0]),
    ((40, 24, 23), 300, 3, None),
]


@pytest.mark.parametrize("precision", [hs.HS_BF16, hs.HS_FP32_CHECK])
@pytest.mark.parametrize("dims,N,M,weights", EDGE)
def test_edge_shapes(dims, N, M, weights, precision):
    rng = np.random.default_rng(len(dims) * 100 + N)
    x = rng.standard_normal((N, dims[0]), dtype=np.float32)
    y = rng.integers(0, dims[-1], N, dtype=np.int32)
    theta0 = synth.he_normal_params(synth.MLP, dims, 7)
    theta0[theta0.size - dims[-1]:] = rng.standard_normal(dims[-1]).astype(np.float32) * 0.1   # nonzero last bias
    for sync in (hs.HS_SYNC_MEAN, hs.HS_SYNC_CP_WEIGHTED):
        lib = run_library(synth.MLP, dims, M, N, weights, x, y, theta0, 0.05, 10, precision, sync)
        orc = run_oracle(synth.MLP, dims, M, N, weights, x, y, theta0, 0.05, 10, sync, decide=decide_for(precision))
        _check(lib, orc, theta0.astype(np.float64), precision, 10)


def test_slabs_are_per_worker_gradients():
    wl = synth.WORKLOADS[synth.CFG2]
    x, y = synth.make_batch(wl)
    theta0 = synth.make_params(wl)
    w = synth.initial_weights(wl)
    for precision in (hs.HS_FP32_CHECK, hs.HS_BF16):
        lib = run_library(wl.arch, wl.dims, wl.workers, wl.global_batch, w, x, y, theta0, wl.lr, 1, precision,
                          hs.HS_SYNC_MEAN, keep_slabs=True)
        orc = run_oracle(wl.arch, wl.dims, wl.workers, wl.global_batch, w, x, y, theta0, wl.lr, 1,
                         hs.HS_SYNC_MEAN, keep_slabs=True, decide=decide_for(precision))
        for m in range(wl.workers):
            assert rel(lib["slabs_first"][m], orc["slabs_first"][m]) <= TOL_G[precision], m


@pytest.mark.parametrize("dims,N,M", [((13, 7, 5), 11, 3), ((3, 2), 4, 2), ((50, 33, 17, 2), 97, 6)])
def test_fp32_check_path_odd_widths(dims, N, M):
    rng = np.random.default_rng(N)
    x = rng.standard_normal((N, dims[0]), dtype=np.float32)
    y = rng.integers(0, dims[-1], N, dtype=np.int32)
    theta0 = synth.he_normal_params(synth.MLP, dims, 3)
    w = list(rng.uniform(0.5, 2.0, M))
    lib = run_library(synth.MLP, dims, M, N, w, x, y, theta0, 0.1, 10, hs.HS_FP32_CHECK, hs.HS_SYNC_CP_WEIGHTED)
    orc = run_oracle(synth.MLP, dims, M, N, w, x, y, theta0, 0.1, 10, hs.HS_SYNC_CP_WEIGHTED,
                     decide=decide_for(hs.HS_FP32_CHECK))
    _check(lib, orc, theta0.astype(np.float64), hs.HS_FP32_CHECK, 10)


def test_bf16_rejects_unaligned_widths():
    with pytest.raises(hs.HsError) as e:
        hs.hs_init(synth.MLP, (13, 7, 5), 2, 8, precision=hs.HS_BF16)
    assert e.value.status == hs.HS_ERR_UNSUPPORTED


# The first-step gradient against the oracle with exact (fp64) ReLU' decisions differs by the kink
# flips that bf16 operand rounding causes.  The bounds come from the CPU emulation of the bf16
# arithmetic (tests/bf16_emulation.py: RECORDED holds how far it lands from the exact-decision
# oracle on the same step, BOUND_VS_EXACT_DECISIONS sits at least 1.4x above).  The
# 4096-8192-8192-1000 workload's two smallest workers are checked in
# test_gpu_step_behaviour.test_headline_workload_sampled_parity.
EXACT_DECISION_GAP = [synth.CFG1, synth.CFG2, synth.CFG3, synth.CFG4]


@pytest.mark.parametrize("name", EXACT_DECISION_GAP)
def test_bf16_against_exact_decisions(name):
    wl, x, y, theta0, w = _inputs(name)
    if wl.weight_kind == "drift":
        w = None                       # the drifting workload starts from the even split
    lib = run_library(wl.arch, wl.dims, wl.workers, wl.global_batch, w, x, y, theta0, wl.lr, 1, hs.HS_BF16,
                      hs.HS_SYNC_CP_WEIGHTED)
    orc = run_oracle(wl.arch, wl.dims, wl.workers, wl.global_batch, w, x, y, theta0, wl.lr, 1,
                     hs.HS_SYNC_CP_WEIGHTED)
    assert rel(lib["g_first"], orc["g_first"]) <= BOUND_VS_EXACT_DECISIONS[name]


# ------------------------------------------------------------------------------------------ CNN
@pytest.mark.parametrize("precision,steps", [(hs.HS_BF16, 10), (hs.HS_FP32_CHECK, 3)])
def test_cnn_workload(precision, steps):
    """CNN 3x32x32 -> conv64 -> conv128/2 -> conv256/2 -> pool -> fc10, N = 512, M = 4 (1:2:3:6)."""
    wl, x, y, theta0, w = _inputs(synth.CFG4)
    lib = run_library(wl.arch, wl.dims, wl.workers, wl.global_batch, w, x, y, theta0, wl.lr, steps, precision,
                      hs.HS_SYNC_CP_WEIGHTED, keep_slabs=True)
    orc = run_oracle(wl.arch, wl.dims, wl.workers, wl.global_batch, w, x, y, theta0, wl.lr, steps,
                     hs.HS_SYNC_CP_WEIGHTED, keep_slabs=True, decide=decide_for(precision))
    assert lib["counts"][0] == [43, 85, 128, 256]
    _check(lib, orc, theta0.astype(np.float64), precision, steps)
    for m in range(wl.workers):
        assert rel(lib["slabs_first"][m], orc["slabs_first"][m]) <= TOL_G[precision], m


CNN_EDGE = [
    # Cin, H, W, c1, c2, c3, classes; N; M; weights (odd spatial sizes, one sample per worker)
    ((3, 9, 7, 8, 16, 24, 5), 7, 3, [1.0, 2.0, 4.0]),
    ((2, 6, 6, 16, 8, 8, 3), 4, 4, None),
    ((3, 16, 16, 32, 32, 64, 10), 33, 2, [1.0, 5.0]),
    # implicit patch rows (bf16): 8x8 and 4x4 output grids (several images per 64-row block), 13 images
    ((3, 16, 16, 64, 128, 64, 7), 13, 3, [1.0, 2.0, 3.5]),
    # 8x16 and 4x8 output grids, two workers
    ((3, 16, 32, 64, 64, 64, 5), 9, 2, [2.0, 1.0]),
    # 15x15 input: conv 2 implicit but with an odd input grid (patch-space input gradient), conv 3
    # implicit and sub-pixel
    ((3, 15, 15, 64, 128, 64, 6), 11, 3, [1.0, 1.0, 3.0]),
    # 36 workers: weight-gradient plans over two launches, split-K parts bounded by the smallest worker
    ((3, 16, 16, 64, 128, 64, 7), 40, 36, None),
]


@pytest.mark.parametrize("precision", [hs.HS_BF16, hs.HS_FP32_CHECK])
@pytest.mark.parametrize("dims,N,M,weights", CNN_EDGE)
def test_cnn_edge_shapes(dims, N, M, weights, precision):
    rng = np.random.default_rng(N + dims[1])
    x = rng.standard_normal((N,) + tuple(dims[:3]), dtype=np.float32)
    y = rng.integers(0, dims[-1], N, dtype=np.int32)
    theta0 = synth.he_normal_params(synth.CNN, dims, 5)
    for sync in (hs.HS_SYNC_MEAN, hs.HS_SYNC_CP_WEIGHTED):
        lib = run_library(synth.CNN, dims, M, N, weights, x, y, theta0, 0.05, 10, precision, sync)
        orc = run_oracle(synth.CNN, dims, M, N, weights, x, y, theta0, 0.05, 10, sync, decide=decide_for(precision))
        _check(lib, orc, theta0.astype(np.float64), precision, 10)


# ------------------------------------------------------------------ the Section 5 training recipe
@pytest.mark.parametrize("name,precision", [(synth.CFG2, hs.HS_BF16), (synth.CFG2, hs.HS_FP32_CHECK),
                                            (synth.CFG4, hs.HS_BF16), (synth.CFG1, hs.HS_BF16)])
def test_momentum_weight_decay_cosine_lr(name, precision):
    """SGD momentum 0.9, weight decay 5e-4, cosine-annealed learning rate over the 10 steps."""
    wl, x, y, theta0, w = _inputs(name)
    recipe = (0.9, 5e-4)
    sched = lambda t: hs.hs_cosine_lr(wl.lr, 0.0, t, 10)   # noqa: E731
    lib = run_library(wl.arch, wl.dims, wl.workers, wl.global_batch, w, x, y, theta0, sched, 10, precision,
                      hs.HS_SYNC_CP_WEIGHTED, recipe=recipe)
    orc = run_oracle(wl.arch, wl.dims, wl.workers, wl.global_batch, w, x, y, theta0, sched, 10,
                     hs.HS_SYNC_CP_WEIGHTED, decide=decide_for(precision), recipe=recipe)
    _check(lib, orc, theta0.astype(np.float64), precision, 10)


# ------------------------------------------------------------------ slab-free formulation
@pytest.mark.parametrize("name,precision,sync", [(synth.CFG1, hs.HS_BF16, hs.HS_SYNC_CP_WEIGHTED),
                                                 (synth.CFG2, hs.HS_BF16, hs.HS_SYNC_MEAN),
                                                 (synth.CFG2, hs.HS_FP32_CHECK, hs.HS_SYNC_CP_WEIGHTED),
                                                 (synth.CFG2, hs.HS_FP32_CHECK, hs.HS_SYNC_MEAN)])
def test_fused_sync_matches_oracle(name, precision, sync):
    """sum_m w_m G_m as one all-rows product with the weights folded into the loss-gradient scale."""
    wl, x, y, theta0, w = _inputs(name)
    lib = run_library(wl.arch, wl.dims, wl.workers, wl.global_batch, w, x, y, theta0, wl.lr, 10, precision, sync,
                      fused=True)
    orc = _oracle_run(name, sync, 10, precision)
    _check(lib, orc, theta0.astype(np.float64), precision, 10)


def test_fused_sync_headline_workload_gradient():
    """4096-8192-8192-1000, N 16384, M 16: the slab-free gradient equals the slab gradient (same kernels,
    different summation order) and the step keeps working with the per-worker losses."""
    wl, x, y, theta0, w = _inputs(synth.CFG5)
    a = run_library(wl.arch, wl.dims, wl.workers, wl.global_batch, w, x, y, theta0, wl.lr, 1, hs.HS_BF16,
                    hs.HS_SYNC_CP_WEIGHTED)
    b = run_library(wl.arch, wl.dims, wl.workers, wl.global_batch, w, x, y, theta0, wl.lr, 1, hs.HS_BF16,
                    hs.HS_SYNC_CP_WEIGHTED, fused=True)
    assert rel(b["g_first"], a["g_first"]) <= 5e-3
    assert a["worker_losses_first"] == b["worker_losses_first"]


# ------------------------------------------------------------------ implicit-GEMM convolutions
def _cnn_run(monkeypatch, mode, wl, x, y, theta0, w, steps):
    monkeypatch.setenv("HS_CONV_IMPLICIT", mode)
    torch.cuda.synchronize()
    free0 = torch.cuda.mem_get_info()[0]
    ctx = hs.hs_init(wl.arch, wl.dims, wl.workers, wl.global_batch, compute_weights=w, precision=hs.HS_BF16)
    used = free0 - torch.cuda.mem_get_info()[0]
    try:
        hs.hs_set_debug(ctx, True)
        p = torch.tensor(theta0, device="cuda")
        xd, yd = torch.from_numpy(x).cuda(), torch.from_numpy(y).cuda()
        losses, first = [], None
        for t in range(steps):
            losses.append(hs.hs_step(ctx, p, xd, yd, None, wl.lr))
            if t == 0:
                first = torch.empty(wl.workers, ctx.P, device="cuda")
                hs.hs_debug_grads(ctx, None, first)
        torch.cuda.synchronize()
        return p.cpu(), losses, first.cpu(), used
    finally:
        ctx.close()


def test_implicit_conv_is_bit_identical_to_materialised_patches(monkeypatch):
    """The convolutions' forward and weight-gradient products read their patch rows straight from the
    NHWC input (4-D TMA boxes; HS_CONV_IMPLICIT=fwd) or from materialised patch rows
    (HS_CONV_IMPLICIT=0): same operand values in the same k-block order, so theta, losses and
    per-worker gradients agree bit for bit, and the implicit context holds no patch buffers for the
    second and third convolutions."""
    wl, x, y, theta0, w = _inputs(synth.CFG4)
    imp = _cnn_run(monkeypatch, "fwd", wl, x, y, theta0, w, 3)
    mat = _cnn_run(monkeypatch, "0", wl, x, y, theta0, w, 3)
    assert torch.equal(imp[0], mat[0])
    assert imp[1] == mat[1]
    assert torch.equal(imp[2], mat[2])
    n = wl.global_batch
    saved = 2 * (n * 256 * 584 + n * 64 * 1160)      # bf16 patch rows of conv2 and conv3
    assert mat[3] - imp[3] >= 0.9 * saved


def test_subpixel_input_gradient_matches_patch_space_gather(monkeypatch):
    """The stride-2 convolutions' input gradients as four grouped sub-pixel products (default) against
    the patch-space product followed by the gather (HS_CONV_IMPLICIT=fwd): the same sums in another
    fp32 order, rounded to bf16 once, so first-step gradients agree to bf16 rounding and the
    patch-space buffer (fp32 N*16*16 x 576) is gone."""
    wl, x, y, theta0, w = _inputs(synth.CFG4)
    sub = _cnn_run(monkeypatch, "1", wl, x, y, theta0, w, 3)
    pat = _cnn_run(monkeypatch, "fwd", wl, x, y, theta0, w, 3)
    assert rel(sub[2].numpy(), pat[2].numpy()) <= 2e-3
    assert np.allclose(sub[1], pat[1], rtol=1e-3, atol=0)
    assert rel(sub[0].numpy(), pat[0].numpy()) <= 1e-5
    assert pat[3] - sub[3] >= 0.9 * 4 * wl.global_batch * 256 * 576


def _cnn_run_env(monkeypatch, env, wl, x, y, theta0, w, steps):
    for k, v in env.items():
        monkeypatch.setenv(k, v)
    try:
        return _cnn_run(monkeypatch, "1", wl, x, y, theta0, w, steps)
    finally:
        for k in env:
            monkeypatch.delenv(k)


@pytest.mark.parametrize("dims,N,M", [(None, None, None), ((3, 16, 16, 64, 128, 64, 7), 13, 3)])
def test_conv_a_boxes_of_128_pixels_are_bit_identical(monkeypatch, dims, N, M):
    """One 128-pixel 4-D box per 128 rows of the convolutions' A operands (forward patch rows,
    shifted sub-pixel output gradient) lands in shared memory exactly as two 64-pixel boxes do, so
    theta, losses and per-worker gradients agree bit for bit with HS_CONV_ABOX=64 (the CNN workload,
    and 8x8 / 4x4 output grids where a box spans two or eight images, with a ragged last image)."""
    if dims is None:
        wl, x, y, theta0, w = _inputs(synth.CFG4)
    else:
        rng = np.random.default_rng(3)
        x = rng.standard_normal((N,) + tuple(dims[:3]), dtype=np.float32)
        y = rng.integers(0, dims[-1], N, dtype=np.int32)
        theta0 = synth.he_normal_params(synth.CNN, dims, 5)
        wl = types.SimpleNamespace(arch=synth.CNN, dims=dims, global_batch=N, workers=M, lr=0.05)
        w = [1.0, 2.0, 3.5]
    big = _cnn_run_env(monkeypatch, {}, wl, x, y, theta0, w, 3)
    small = _cnn_run_env(monkeypatch, {"HS_CONV_ABOX": "64"}, wl, x, y, theta0, w, 3)
    assert torch.equal(big[0], small[0])
    assert big[1] == small[1]
    assert torch.equal(big[2], small[2])


def _env_run(monkeypatch, env, fn):
    for k, v in env.items():
        monkeypatch.setenv(k, v)
    try:
        return fn()
    finally:
        for k in env:
            monkeypatch.delenv(k)


@pytest.mark.parametrize("case", ["cnn", "mlp_ragged", "mlp_tile_averaged"])
def test_two_kblocks_per_stage_are_bit_identical(monkeypatch, case):
    """Two k-blocks per pipeline stage (one barrier round trip feeding two k-blocks of MMAs) issue the
    same MMAs on the same operands in the same order as one, so every result is the same bit for
    bit: the CNN workload (default: two for every convolution product and 256 x 128 tile, against
    HS_KSTAGE=1), and an MLP with ragged worker segments whose grouped weight gradients end in
    partial k-blocks and odd k-block counts (HS_KSTAGE=2 against 1); the same MLP stepped as users
    step it (no read-back, every layer's weight gradient on the tile-averaged kernel: the forward
    products take two k-blocks per stage by default, against HS_KSTAGE=1)."""
    if case == "cnn":
        wl, x, y, theta0, w = _inputs(synth.CFG4)
        args = (wl.arch, wl.dims, wl.workers, wl.global_batch, w, x, y, theta0, wl.lr, 3)
        env_a, env_b = {}, {"HS_KSTAGE": "1"}
    else:
        dims, N, M, w = (256, 192, 136, 10), 333, 3, [1.0, 2.0, 3.5]
        rng = np.random.default_rng(11)
        x = rng.standard_normal((N, dims[0]), dtype=np.float32)
        y = rng.integers(0, dims[-1], N, dtype=np.int32)
        theta0 = synth.he_normal_params(synth.MLP, dims, 4)
        args = (synth.MLP, dims, M, N, w, x, y, theta0, 0.05, 3)
        env_a, env_b = {"HS_KSTAGE": "2"}, {"HS_KSTAGE": "1"}
        if case == "mlp_tile_averaged":
            env_a, env_b = {"HS_TILE_AVERAGE": "all"}, {"HS_TILE_AVERAGE": "all", "HS_KSTAGE": "1"}
    debug = case != "mlp_tile_averaged"

    def go():
        return run_library(*args, hs.HS_BF16, hs.HS_SYNC_CP_WEIGHTED, keep_slabs=debug, debug=debug)

    a = _env_run(monkeypatch, env_a, go)
    b = _env_run(monkeypatch, env_b, go)
    assert np.array_equal(a["theta"], b["theta"])
    assert a["losses"] == b["losses"]
    if debug:
        assert np.array_equal(a["slabs_first"], b["slabs_first"])


@pytest.mark.parametrize("dims,N,M,weights", [(None, None, None, None),
                                              ((3, 9, 7, 8, 16, 24, 5), 7, 3, [1.0, 2.0, 4.0]),
                                              ((2, 6, 6, 16, 8, 8, 3), 4, 4, None),
                                              ((3, 16, 16, 32, 32, 64, 10), 33, 2, [1.0, 5.0])])
def test_first_convolution_kernel_is_bit_identical(monkeypatch, dims, N, M, weights):
    """The first convolution's forward as one kernel (patch rows built in shared memory from the NCHW
    input and written out for the weight gradient, resident weights, bias + ReLU) against the
    materialised patch rows and the tiled product (HS_CONV_FIRST=0): same bf16 operands and fp32
    sums, so theta, losses and per-worker gradients agree bit for bit - on the CNN workload and on
    8-, 16- and 32-channel first convolutions over odd grids with a ragged last tile."""
    if dims is None:
        wl, x, y, theta0, w = _inputs(synth.CFG4)
    else:
        rng = np.random.default_rng(N + dims[1])
        x = rng.standard_normal((N,) + tuple(dims[:3]), dtype=np.float32)
        y = rng.integers(0, dims[-1], N, dtype=np.int32)
        theta0 = synth.he_normal_params(synth.CNN, dims, 5)
        wl = types.SimpleNamespace(arch=synth.CNN, dims=dims, global_batch=N, workers=M, lr=0.05)
        w = weights
    one = _cnn_run_env(monkeypatch, {}, wl, x, y, theta0, w, 3)
    two = _cnn_run_env(monkeypatch, {"HS_CONV_FIRST": "0"}, wl, x, y, theta0, w, 3)
    assert torch.equal(one[0], two[0])
    assert one[1] == two[1]
    assert torch.equal(one[2], two[2])


@pytest.mark.parametrize("dims,N,M,weights", [(None, None, None, None),
                                              ((3, 16, 16, 64, 128, 64, 7), 13, 3, [1.0, 2.0, 3.5]),
                                              ((3, 16, 32, 64, 64, 64, 5), 9, 2, [2.0, 1.0])])
def test_subpixel_one_product_is_bit_identical(monkeypatch, dims, N, M, weights):
    """The stride-2 convolutions' input gradients as one product over the four sub-pixel classes
    (columns in four class blocks, the four shifts of the output gradient as K, zero weight blocks
    where a class has no tap with that shift) against one grouped product per class
    (HS_SUBPIXEL=classes): every class sums the same products in the same order with exact zeros
    between, so theta, losses and per-worker gradients agree bit for bit - on the CNN workload, and on
    8x8 / 4x4 and 8x16 / 4x8 output grids with 64- and 128-channel inputs."""
    if dims is None:
        wl, x, y, theta0, w = _inputs(synth.CFG4)
    else:
        rng = np.random.default_rng(N + dims[1])
        x = rng.standard_normal((N,) + tuple(dims[:3]), dtype=np.float32)
        y = rng.integers(0, dims[-1], N, dtype=np.int32)
        theta0 = synth.he_normal_params(synth.CNN, dims, 5)
        wl = types.SimpleNamespace(arch=synth.CNN, dims=dims, global_batch=N, workers=M, lr=0.05)
        w = weights
    one = _cnn_run_env(monkeypatch, {}, wl, x, y, theta0, w, 3)
    grouped = _cnn_run_env(monkeypatch, {"HS_SUBPIXEL": "classes"}, wl, x, y, theta0, w, 3)
    assert torch.equal(one[0], grouped[0])
    assert one[1] == grouped[1]
    assert torch.equal(one[2], grouped[2])


@pytest.mark.parametrize("dims,N,M,weights", [(None, None, None, None),
                                              ((3, 16, 16, 64, 128, 64, 7), 13, 3, [1.0, 2.0, 3.5])])
@pytest.mark.parametrize("subpixel", ["", "classes"])
def test_cnn_relu_bits_are_bit_identical(monkeypatch, dims, N, M, weights, subpixel):
    """ReLU' of the first two convolutions' activations stored as bits by their forward epilogues and
    read by the next convolution's sub-pixel input gradient at its class pixels, against reading the
    bf16 activations themselves (HS_RELU_BITS=0): the same decisions, so the same bits everywhere,
    for the one-product and the per-class sub-pixel forms."""
    if dims is None:
        wl, x, y, theta0, w = _inputs(synth.CFG4)
    else:
        rng = np.random.default_rng(N + dims[1])
        x = rng.standard_normal((N,) + tuple(dims[:3]), dtype=np.float32)
        y = rng.integers(0, dims[-1], N, dtype=np.int32)
        theta0 = synth.he_normal_params(synth.CNN, dims, 5)
        wl = types.SimpleNamespace(arch=synth.CNN, dims=dims, global_batch=N, workers=M, lr=0.05)
        w = weights
    env = {"HS_SUBPIXEL": subpixel} if subpixel else {}
    bits = _cnn_run_env(monkeypatch, env, wl, x, y, theta0, w, 3)
    acts = _cnn_run_env(monkeypatch, dict(env, HS_RELU_BITS="0"), wl, x, y, theta0, w, 3)
    assert torch.equal(bits[0], acts[0])
    assert bits[1] == acts[1]
    assert torch.equal(bits[2], acts[2])
