"""hs_step's own CUDA graph of the step: after one eager step a context captures its step per key
(parameters, inputs, momentum state, profiling) and replays it, with the learning rate written to
device memory ahead of each replay.  Replayed steps must equal eager steps (HS_STEP_GRAPH=0) bit
for bit, through learning-rate changes, repartitions, debug read-back, the momentum recipe, staged
inputs and profiling; and the per-phase profile keeps its events and launch counts."""
import numpy as np
import pytest
import torch

import synth
import paper_2110_08941_gb300 as hs

pytestmark = pytest.mark.gpu


def _run(monkeypatch, graph, wl, x, y, theta0, w, precision, steps, lr_of, repartition=None, recipe=None,
         debug_at=(), profile_at=(), staged=False):
    monkeypatch.setenv("HS_STEP_GRAPH", "1" if graph else "0")
    ctx = hs.hs_init(wl.arch, wl.dims, wl.workers, wl.global_batch, compute_weights=w, precision=precision)
    try:
        if recipe:
            hs.hs_set_optimizer(ctx, *recipe)
        p = torch.tensor(theta0, device="cuda")
        xd, yd = torch.from_numpy(x).cuda(), torch.from_numpy(y).cuda()
        xh, yh = torch.from_numpy(x).pin_memory(), torch.from_numpy(y).pin_memory()
        losses, grads, prof = [], [], []
        for t in range(steps):
            if repartition and t in repartition:
                hs.hs_partition(ctx, repartition[t])
            hs.hs_set_debug(ctx, t in debug_at)
            hs.hs_set_profiling(ctx, t in profile_at)
            if staged:
                losses.append(hs.hs_step(ctx, p, hs.hs_stage_inputs(ctx, xh, yh), None, None, lr_of(t)))
            else:
                losses.append(hs.hs_step(ctx, p, xd, yd, None, lr_of(t)))
            if t in debug_at:
                g = torch.empty(ctx.P, device="cuda")
                hs.hs_debug_grads(ctx, g, None)
                grads.append(g.cpu())
            if t in profile_at:
                prof.append(hs.hs_read_profile(ctx))
        torch.cuda.synchronize()
        return p.cpu(), losses, grads, prof
    finally:
        ctx.close()


CASES = [
    # name, precision, recipe, staged
    (synth.CFG1, hs.HS_BF16, None, False),
    (synth.CFG2, hs.HS_BF16, (0.9, 5e-4), False),
    (synth.CFG2, hs.HS_FP32_CHECK, None, True),
    (synth.CFG3, hs.HS_BF16, None, False),
    (synth.CFG4, hs.HS_BF16, (0.9, 5e-4), True),
]


@pytest.mark.parametrize("name,precision,recipe,staged", CASES)
def test_replayed_steps_equal_eager_steps(monkeypatch, name, precision, recipe, staged):
    wl = synth.WORKLOADS[name]
    x, y = synth.make_batch(wl)
    theta0 = synth.make_params(wl)
    w = synth.initial_weights(wl)
    steps = 9
    lr_of = lambda t: hs.hs_cosine_lr(wl.lr, 0.0, t, steps)   # noqa: E731  (a new lr every step)
    rng = np.random.default_rng(5)
    rep = {5: list(rng.uniform(0.5, 2.0, wl.workers))}
    kw = dict(repartition=rep, recipe=recipe, debug_at=(3,), profile_at=(1, 2, 6, 7), staged=staged)
    a = _run(monkeypatch, True, wl, x, y, theta0, w, precision, steps, lr_of, **kw)
    b = _run(monkeypatch, False, wl, x, y, theta0, w, precision, steps, lr_of, **kw)
    assert torch.equal(a[0], b[0])
    assert a[1] == b[1]
    for ga, gb in zip(a[2], b[2]):
        assert torch.equal(ga, gb)
    # the profile of a replayed step: every phase timed, the same kernels counted (plus the one that
    # writes the learning rate, counted with the update)
    assert len(a[3]) == len(b[3]) == 4
    for (pa, pb) in zip(a[3], b[3]):
        for phase in pa:
            ms_a, n_a = pa[phase]
            ms_b, n_b = pb[phase]
            # launch counts run over the unprofiled steps since the last read as well, times only
            # over the profiled step: compare the two modes with each other
            assert (ms_a > 0) == (ms_b > 0), phase
            extra = 1 if phase == "update" and n_a != n_b else 0
            assert n_a == n_b + extra, (phase, n_a, n_b)
