"""The tile-averaged weight-gradient launch: each worker's weight gradient g^m (Eq. 1) formed tile
by tile in tensor memory, averaged in worker order (Section 1; Section 4.2's weights) and applied to
theta in the same kernel.  It must leave theta and the bf16 weight copy exactly where the slab path
(per-worker gradients stored, then reduce_update_kernel) leaves them, and within the oracle's
tolerance, over several steps, repartitions, worker counts, sync rules and ragged shapes."""
import os

import numpy as np
import pytest
import torch

import synth
import paper_2110_08941_gb300 as hs
from tests.gpu_helpers import decide_for, rel, run_library, run_oracle

pytestmark = pytest.mark.gpu


def _init(dims, M, N, weights, sync, tile):
    old = os.environ.get("HS_TILE_AVERAGE")
    os.environ["HS_TILE_AVERAGE"] = "all" if tile else "0"
    try:
        return hs.hs_init(hs.HS_MLP, dims, M, N, compute_weights=weights, sync=sync)
    finally:
        if old is None:
            os.environ.pop("HS_TILE_AVERAGE")
        else:
            os.environ["HS_TILE_AVERAGE"] = old


def _run(dims, M, N, weights, sync, tile, steps, lr, x, y, theta0, repartition=None, recipe=None):
    ctx = _init(dims, M, N, weights, sync, tile)
    try:
        if recipe is not None:
            hs.hs_set_optimizer(ctx, *recipe)
        p = torch.tensor(theta0, device="cuda")
        xd, yd = torch.from_numpy(x).cuda(), torch.from_numpy(y).cuda()
        losses = []
        for t in range(steps):
            if repartition is not None and t in repartition:
                hs.hs_partition(ctx, repartition[t])
            losses.append(hs.hs_step(ctx, p, xd, yd, None, lr))
        # one more forward pass reads the bf16 weight copy the last update wrote
        losses.append(hs.hs_step(ctx, p, xd, yd, None, 0.0))
        torch.cuda.synchronize()
        return p.cpu(), losses
    finally:
        ctx.close()


def _data(dims, N, seed):
    wl = synth.Workload("t", synth.MLP, tuple(dims), dims[-1], N, 1, (1.0,), 1, 0.0, seed=seed)
    x, y = synth.make_batch(wl)
    return np.ascontiguousarray(x), np.ascontiguousarray(y), synth.he_normal_params(synth.MLP, dims, seed)


CASES = [
    # dims, N, M, compute weights, sync
    ((3072, 1024, 1024, 10), 1024, 4, (1.0, 1.0, 2.0, 4.0), hs.HS_SYNC_CP_WEIGHTED),
    ((3072, 1024, 1024, 10), 1024, 4, (1.0, 1.0, 2.0, 4.0), hs.HS_SYNC_MEAN),
    ((3072, 1024, 1024, 10), 1024, 4, (1.0, 1.0, 2.0, 4.0), hs.HS_SYNC_CP_LITERAL),
    # ragged: widths not multiples of the 256-wide tile, worker rows not multiples of 64
    ((264, 200, 136, 10), 300, 5, (1.0, 2.0, 3.0, 1.5, 0.7), hs.HS_SYNC_CP_WEIGHTED),
    # 1000 classes (partial last row tile), 16 lognormal workers
    ((512, 768, 1000), 2048, 16, tuple(synth.lognormal_weights(16, 3)), hs.HS_SYNC_CP_WEIGHTED),
    # the most groups one launch takes
    ((256, 512, 10), 2048, 32, tuple(np.linspace(0.5, 2.0, 32)), hs.HS_SYNC_MEAN),
    # one worker; a worker left with a single sample
    ((256, 512, 10), 512, 1, (1.0,), hs.HS_SYNC_MEAN),
    ((256, 512, 10), 96, 4, (1e-6, 1.0, 1.0, 1.0), hs.HS_SYNC_CP_WEIGHTED),
    # more workers than one launch takes: the slab path on both sides
    ((256, 512, 10), 2048, 33, tuple(np.linspace(0.5, 2.0, 33)), hs.HS_SYNC_CP_WEIGHTED),
]


@pytest.mark.parametrize("dims,N,M,weights,sync", CASES)
def test_tile_average_equals_slab_path(dims, N, M, weights, sync):
    x, y, theta0 = _data(dims, N, seed=11)
    rep = {2: tuple(reversed(weights))} if M > 1 else None
    a, la = _run(dims, M, N, weights, sync, True, 4, 0.05, x, y, theta0, rep)
    b, lb = _run(dims, M, N, weights, sync, False, 4, 0.05, x, y, theta0, rep)
    assert torch.equal(a, b)
    assert la == lb
    assert not torch.equal(a, torch.from_numpy(theta0))


@pytest.mark.parametrize("dims,N,M,weights", [((3072, 1024, 1024, 10), 1024, 4, (1.0, 1.0, 2.0, 4.0)),
                                               ((264, 200, 136, 10), 300, 5, (1.0, 2.0, 3.0, 1.5, 0.7))])
def test_tile_average_with_momentum_equals_slab_path(dims, N, M, weights):
    """The experiments' optimiser (Section 5: momentum 0.9, weight decay 5e-4) in the tile kernel's
    epilogue: the momentum buffer starts as d on the first step and both forms agree bit for bit."""
    x, y, theta0 = _data(dims, N, seed=13)
    rep = {3: tuple(reversed(weights))}
    a, la = _run(dims, M, N, weights, hs.HS_SYNC_CP_WEIGHTED, True, 5, 0.05, x, y, theta0, rep, (0.9, 5e-4))
    b, lb = _run(dims, M, N, weights, hs.HS_SYNC_CP_WEIGHTED, False, 5, 0.05, x, y, theta0, rep, (0.9, 5e-4))
    assert torch.equal(a, b)
    assert la == lb


def test_tile_average_momentum_matches_oracle(monkeypatch):
    """Momentum 0.9, weight decay 5e-4 and a cosine learning rate over 10 steps through the tile
    kernel (no debug read-back), against the oracle's recipe."""
    monkeypatch.setenv("HS_TILE_AVERAGE", "all")
    wl = synth.WORKLOADS[synth.CFG2]
    x, y = synth.make_batch(wl)
    theta0 = synth.make_params(wl)
    weights = synth.initial_weights(wl)
    recipe = (0.9, 5e-4)
    sched = lambda t: hs.hs_cosine_lr(wl.lr, 0.0, t, 10)   # noqa: E731
    lib = run_library(wl.arch, wl.dims, wl.workers, wl.global_batch, weights, x, y, theta0, sched, 10,
                      hs.HS_BF16, hs.HS_SYNC_CP_WEIGHTED, recipe=recipe, debug=False)
    orc = run_oracle(wl.arch, wl.dims, wl.workers, wl.global_batch, weights, x, y, theta0, sched, 10,
                     hs.HS_SYNC_CP_WEIGHTED, decide=decide_for(hs.HS_BF16), recipe=recipe)
    assert rel(lib["theta"], orc["theta"]) <= 2e-2
    assert rel(lib["theta"] - theta0, orc["theta"] - theta0) <= 5e-2


@pytest.mark.parametrize("name", [synth.CFG2, synth.CFG3])
def test_tile_average_matches_oracle(name, monkeypatch):
    monkeypatch.setenv("HS_TILE_AVERAGE", "all")   # every layer, however few its weight tiles
    wl = synth.WORKLOADS[name]
    x, y = synth.make_batch(wl)
    theta0 = synth.make_params(wl)
    weights = synth.initial_weights(wl)
    steps = 3
    lib = run_library(wl.arch, wl.dims, wl.workers, wl.global_batch, weights, x, y, theta0, wl.lr, steps,
                      hs.HS_BF16, hs.HS_SYNC_CP_WEIGHTED, debug=False)
    orc = run_oracle(wl.arch, wl.dims, wl.workers, wl.global_batch, weights, x, y, theta0, wl.lr, steps,
                     hs.HS_SYNC_CP_WEIGHTED, decide=decide_for(hs.HS_BF16))
    d_lib = lib["theta"] - theta0
    d_orc = orc["theta"] - theta0
    assert rel(lib["theta"], orc["theta"]) <= 2e-2
    assert rel(d_lib, d_orc) <= 5e-2
    assert np.allclose(lib["losses"], orc["losses"], rtol=2e-2)


def test_tile_average_full_size_equals_slab_path():
    """The 4096-8192-8192-1000 workload (N 16384, 16 workers): two steps on each path, theta equal
    bit for bit."""
    wl = synth.WORKLOADS[synth.CFG5]
    x, y = synth.make_batch(wl)
    theta0 = synth.make_params(wl)
    weights = tuple(synth.initial_weights(wl))
    a, la = _run(wl.dims, wl.workers, wl.global_batch, weights, hs.HS_SYNC_CP_WEIGHTED, True, 2, wl.lr,
                 x, y, theta0)
    b, lb = _run(wl.dims, wl.workers, wl.global_batch, weights, hs.HS_SYNC_CP_WEIGHTED, False, 2, wl.lr,
                 x, y, theta0)
    assert torch.equal(a, b)
    assert la == lb


def test_slab_read_back_needs_debug_after_a_tile_step():
    """A step without debug keeps the weight ranges of the per-worker gradients in tensor memory:
    asking for the slabs afterwards is an argument error, and a debug step provides them."""
    dims, N, M = (256, 512, 10), 512, 4
    x, y, theta0 = _data(dims, N, seed=5)
    ctx = _init(dims, M, N, (1.0, 2.0, 3.0, 4.0), hs.HS_SYNC_CP_WEIGHTED, True)
    try:
        p = torch.tensor(theta0, device="cuda")
        xd, yd = torch.from_numpy(x).cuda(), torch.from_numpy(y).cuda()
        hs.hs_step(ctx, p, xd, yd, None, 0.05)
        slabs = torch.empty(M, ctx.P, device="cuda")
        with pytest.raises(hs.HsError):
            hs.hs_debug_grads(ctx, None, slabs)
        hs.hs_set_debug(ctx, True)
        hs.hs_step(ctx, p, xd, yd, None, 0.05)
        hs.hs_debug_grads(ctx, None, slabs)
        torch.cuda.synchronize()
        assert torch.isfinite(slabs).all() and slabs.abs().sum() > 0
    finally:
        ctx.close()


def test_default_takes_the_tile_launch_where_a_layer_fills_the_pairs():
    """Default selection: the tile-averaged launch for layers with at least one 256 x 256 weight
    tile per SM pair, the slab path for the rest, in one step (bit for bit the slab path)."""
    dims, N, M = (256, 4096, 8192, 10), 1024, 4   # layer 2: 32 x 16 tiles (tile launch); 1, 3: slab
    x, y, theta0 = _data(dims, N, seed=9)
    os.environ.pop("HS_TILE_AVERAGE", None)
    ctx = hs.hs_init(hs.HS_MLP, dims, M, N, compute_weights=(1.0, 2.0, 3.0, 4.0))
    try:
        p = torch.tensor(theta0, device="cuda")
        xd, yd = torch.from_numpy(x).cuda(), torch.from_numpy(y).cuda()
        for _ in range(2):
            hs.hs_step(ctx, p, xd, yd, None, 0.05)
        torch.cuda.synchronize()
        with pytest.raises(hs.HsError):   # a tile step: its weight ranges are not in the slabs
            hs.hs_debug_grads(ctx, None, torch.empty(M, ctx.P, device="cuda"))
    finally:
        ctx.close()
    b, _ = _run(dims, M, N, (1.0, 2.0, 3.0, 4.0), hs.HS_SYNC_CP_WEIGHTED, False, 2, 0.05, x, y, theta0)
    assert torch.equal(p.cpu(), b)


def _bf(r, c, g):
    """bf16 [r, c] view of a [r, c rounded up to 8] buffer (16-byte rows), and its fp64 copy."""
    t = (torch.randn(r, (c + 7) // 8 * 8, generator=g, device="cuda") * 0.5).to(torch.bfloat16)[:, :c]
    return t, t.double()


@pytest.mark.parametrize("M,N,groups", [(256, 256, [64]), (300, 520, [1, 63, 64, 65, 200]),
                                        (1000, 512, [242, 2410, 316]), (264, 136, [7] * 32),
                                        (512, 768, [1024, 16, 17, 900])])
def test_kernel_alone_matches_plain_reference(M, N, groups):
    """The kernel through its test hook: theta - lr * sum_g w_g A_g^T B_g against fp64 products of
    the same bf16 operands, over ragged groups (1 row, 63/64/65 rows, 32 groups) and partial
    tiles; the bf16 copy is the rounding of the new theta."""
    g = torch.Generator(device="cuda").manual_seed(M * 7 + N + len(groups))
    K = sum(groups)
    ko = [0]
    for n in groups:
        ko.append(ko[-1] + n)
    A, a = _bf(K, M, g)
    B, b = _bf(K, N, g)
    w = torch.rand(len(groups), generator=g, device="cuda") + 0.5
    theta = torch.randn(M, N, generator=g, device="cuda")
    t0 = theta.double().clone()
    shadow = torch.empty(M, N, device="cuda", dtype=torch.bfloat16)
    lr = 0.03
    hs.hs_debug_wgrad_avg(A, B, ko, w, lr, theta, shadow)
    torch.cuda.synchronize()
    gsum = torch.zeros(M, N, device="cuda", dtype=torch.float64)
    for gi in range(len(groups)):
        gsum += float(w[gi]) * (a[ko[gi]:ko[gi + 1]].t() @ b[ko[gi]:ko[gi + 1]])
    ref = t0 - lr * gsum
    d = theta.double() - t0
    assert float((d - (ref - t0)).norm() / (ref - t0).norm()) < 1e-5
    assert torch.equal(shadow, theta.to(torch.bfloat16))


def test_kernel_alone_bounded_wait_reports_and_leaves_theta():
    """Failure detection without a GPU fault: the kernel's loads are withheld, its bounded waits
    expire, the call reports HS_ERR_DEVICE_CHECK, theta is unchanged and the next call works."""
    g = torch.Generator(device="cuda").manual_seed(3)
    A, _ = _bf(128, 256, g)
    B, _ = _bf(128, 256, g)
    w = torch.ones(2, device="cuda")
    theta = torch.randn(256, 256, generator=g, device="cuda")
    before = theta.clone()
    shadow = torch.empty(256, 256, device="cuda", dtype=torch.bfloat16)
    with pytest.raises(hs.HsError) as e:
        hs.hs_debug_wgrad_avg(A, B, [0, 64, 128], w, 0.1, theta, shadow, test_stall=True)
    assert e.value.status == hs.HS_ERR_DEVICE_CHECK
    assert torch.equal(theta, before)
    hs.hs_debug_wgrad_avg(A, B, [0, 64, 128], w, 0.1, theta, shadow)
    torch.cuda.synchronize()
    assert not torch.equal(theta, before)


@pytest.mark.parametrize("dims,N,M", [((3072, 1024, 1024, 10), 1024, 4), ((264, 200, 136, 10), 300, 5),
                                      ((512, 768, 1000), 2048, 16)])
def test_relu_bits_equal_the_activation_mask(dims, N, M, monkeypatch):
    """The input-gradient products take ReLU' from bits the forward epilogue packs (one per stored
    activation, value > 0); with HS_RELU_BITS=0 they read the bf16 activations: the same decisions,
    so the same parameters bit for bit."""
    x, y, theta0 = _data(dims, N, seed=21)
    weights = tuple(float(v) for v in np.linspace(1.0, 2.0, M))
    out = []
    for bits in ("1", "0"):
        monkeypatch.setenv("HS_RELU_BITS", bits)
        out.append(_run(dims, M, N, weights, hs.HS_SYNC_CP_WEIGHTED, True, 3, 0.05, x, y, theta0))
    assert torch.equal(out[0][0], out[1][0])
    assert out[0][1] == out[1][1]
