"""hs_step inside a CUDA graph: a step captured once (loss not requested) and replayed gives the
same parameters bit for bit as the same number of eager steps."""
import pytest
import torch

import synth
import paper_2110_08941_gb300 as hs

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("name,precision", [(synth.CFG1, hs.HS_BF16), (synth.CFG2, hs.HS_BF16),
                                            (synth.CFG4, hs.HS_BF16), (synth.CFG2, hs.HS_FP32_CHECK)])
def test_captured_step_replays_bit_exact(name, precision):
    wl = synth.WORKLOADS[name]
    x, y = synth.make_batch(wl)
    theta0 = synth.make_params(wl)
    ctx = hs.hs_init(wl.arch, wl.dims, wl.workers, wl.global_batch, compute_weights=synth.initial_weights(wl),
                     precision=precision)
    try:
        xd, yd = torch.from_numpy(x).cuda(), torch.from_numpy(y).cuda()
        ref = torch.tensor(theta0, device="cuda")
        for _ in range(4):
            hs.hs_step(ctx, ref, xd, yd, None, wl.lr, want_loss=False)
        p = torch.tensor(theta0, device="cuda")
        hs.hs_sync_params(ctx, p)
        side = torch.cuda.Stream()
        side.wait_stream(torch.cuda.current_stream())
        with torch.cuda.stream(side):
            hs.hs_step(ctx, p, xd, yd, None, wl.lr, want_loss=False)      # step 1, eager
        torch.cuda.current_stream().wait_stream(side)
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g):
            hs.hs_step(ctx, p, xd, yd, None, wl.lr, want_loss=False)      # recorded, not run
        for _ in range(3):                                                  # steps 2..4
            g.replay()
        torch.cuda.synchronize()
        assert torch.equal(p, ref)
        # the context still steps eagerly afterwards, and reports its loss
        loss = hs.hs_step(ctx, p, xd, yd, None, wl.lr)
        assert loss == loss and loss > 0
    finally:
        ctx.close()
