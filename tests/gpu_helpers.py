"""Shared helpers for the GPU parity tests: run the library through its binding and the oracle
on identical seeded inputs."""
import numpy as np
import torch

import synth
import paper_2110_08941_gb300 as hs
from oracle import cnn, mlp, sgd
from oracle import partition as P

SYNC_TO_ORACLE = {hs.HS_SYNC_MEAN: sgd.SYNC_MEAN, hs.HS_SYNC_CP_WEIGHTED: sgd.SYNC_CP_WEIGHTED,
                  hs.HS_SYNC_CP_LITERAL: sgd.SYNC_CP_LITERAL}


def rel(a, b) -> float:
    a = np.asarray(a, dtype=np.float64)
    b = np.asarray(b, dtype=np.float64)
    return float(np.linalg.norm(a - b) / max(np.linalg.norm(b), 1e-300))


def grad_fn(arch):
    return mlp.worker_loss_grad if arch == synth.MLP else cnn.worker_loss_grad


def _lr_at(lr, t):
    return lr(t) if callable(lr) else lr


def run_library(arch, dims, M, N, weights, x, y, theta0, lr, steps, precision, sync, repartition=None,
                keep_slabs=False, recipe=None, fused=False, debug=True):
    """Returns dict(theta, losses, g_first, slabs_first, counts, index_map).  debug=False runs the
    step as users do (no gradient read-back: the MLP weight gradients take the tile-averaged launch)
    and returns no g_first / slabs_first."""
    ctx = hs.hs_init(arch, dims, M, N, compute_weights=weights, precision=precision, sync=sync)
    try:
        if debug:
            hs.hs_set_debug(ctx, True)
        if recipe is not None:
            hs.hs_set_optimizer(ctx, *recipe)
        if fused:
            hs.hs_set_fused_sync(ctx, True)
        params = torch.tensor(theta0, device="cuda")
        xd = torch.from_numpy(np.ascontiguousarray(x)).cuda()
        yd = torch.from_numpy(np.ascontiguousarray(y)).cuda()
        im = torch.empty(N, dtype=torch.int32, device="cuda")
        part = hs.hs_partition(ctx, index_map_out=im)
        out = dict(losses=[], counts=[list(part.counts)], index_maps=[im.cpu().numpy().copy()])
        for t in range(steps):
            if repartition is not None and t > 0 and t in repartition:
                part = hs.hs_partition(ctx, repartition[t], index_map_out=im)
                out["counts"].append(list(part.counts))
                out["index_maps"].append(im.cpu().numpy().copy())
            out["losses"].append(hs.hs_step(ctx, params, xd, yd, part, _lr_at(lr, t)))
            if t == 0 and debug:
                g = torch.empty(ctx.P, device="cuda")
                slabs = torch.empty(M, ctx.P, device="cuda") if keep_slabs else None
                hs.hs_debug_grads(ctx, g, slabs)
                out["g_first"] = g.cpu().numpy().astype(np.float64)
                out["slabs_first"] = slabs.cpu().numpy().astype(np.float64) if keep_slabs else None
                out["worker_losses_first"] = hs.hs_worker_losses(ctx)
        torch.cuda.synchronize()
        out["theta"] = params.cpu().numpy().astype(np.float64)
        return out
    finally:
        ctx.close()


def decide_for(precision):
    """The kernels take the ReLU' decision from pre-activations of rounded operands (bf16 operands;
    fp32 stored activations with fp64-accumulated forward products on the check path); the oracle
    takes it in the same precision, and every value it computes stays fp64."""
    return mlp.round_bf16 if precision == hs.HS_BF16 else mlp.round_fp32


def run_oracle(arch, dims, M, N, weights, x, y, theta0, lr, steps, sync, repartition=None, keep_slabs=False,
               decide=None, recipe=None):
    fn = grad_fn(arch)
    kw = {} if decide is None else {"decide": decide}
    mode = SYNC_TO_ORACLE[sync]
    cp = list(weights) if weights is not None else [1.0] * M
    sizes = P.partition_sizes(cp, N)
    th = np.asarray(theta0, dtype=np.float64)
    out = dict(losses=[], counts=[list(sizes)])
    buf = None
    for t in range(steps):
        if repartition is not None and t > 0 and t in repartition:
            cp = list(repartition[t])
            sizes = P.partition_sizes(cp, N)
            out["counts"].append(list(sizes))
        lr_t = _lr_at(lr, t)
        th_next, loss, g, slabs, wl = sgd.step(fn, th, dims, x, y, sizes, lr_t, mode,
                                               keep_slabs=(keep_slabs and t == 0), cp=cp, **kw)
        if recipe is None:
            th = th_next
        else:
            th, buf = sgd.momentum_update(th, g, buf if t > 0 else None, lr_t, recipe[0], recipe[1])
        out["losses"].append(loss)
        if t == 0:
            out["g_first"] = g
            out["slabs_first"] = slabs
            out["worker_losses_first"] = wl
    out["theta"] = th
    return out
