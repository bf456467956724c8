"""hs_partition_noalloc: the partition and its device sample->worker map for callers that cannot
allocate device memory (no context; the offsets table lives in a static device array).

Checked against hs_partition, the context-based entry point that computes the same map with
context-owned scratch, and against the oracle's index map (Algorithm 1's sizes, contiguous
segments), on two calls in a row with different compute powers.  The file sorts last
so that a run stopping at the first failure has already run every other test; it also passes
alone in a fresh process (its first call does the per-device set-up)."""
import numpy as np
import pytest
import torch

import paper_2110_08941_gb300 as hs
from oracle import partition as P

pytestmark = pytest.mark.gpu


def test_noalloc_matches_hs_partition_twice():
    M, N = 16, 16384
    ctx = hs.hs_init(hs.HS_MLP, (8, 8, 2), M, N, precision=hs.HS_FP32_CHECK)
    try:
        rng = np.random.default_rng(7)
        for call in range(2):
            cp = list(rng.lognormal(0.0, 0.5 + call, M))
            want_map = torch.full((N,), -1, dtype=torch.int32, device="cuda")
            part = hs.hs_partition(ctx, cp, index_map_out=want_map)
            got_map = torch.full((N,), -7, dtype=torch.int32, device="cuda")
            counts = hs.hs_partition_noalloc(cp, N, got_map)
            torch.cuda.synchronize()
            assert counts == part.counts
            assert torch.equal(got_map, want_map), call
            sizes = P.partition_sizes(cp, N)
            assert counts == sizes
            assert np.array_equal(got_map.cpu().numpy(), np.asarray(P.index_map(sizes), dtype=np.int32)), call
    finally:
        ctx.close()


def test_noalloc_rejects_sizes_beyond_its_table():
    out = torch.empty(4096, dtype=torch.int32, device="cuda")
    with pytest.raises(hs.HsError) as e:
        hs.hs_partition_noalloc([1.0] * 1025, 4096, out)
    assert e.value.status == hs.HS_ERR_INVALID_ARG
    assert "1024" in str(e.value)


def test_noalloc_refuses_bad_output_tensors():
    """A short, int64 or strided device tensor is refused before the library writes through it."""
    for t in (torch.empty(100, dtype=torch.int32, device="cuda"),
              torch.empty(101, dtype=torch.int64, device="cuda"),
              torch.empty(202, dtype=torch.int32, device="cuda")[::2]):
        with pytest.raises(ValueError):
            hs.hs_partition_noalloc([1.0, 3.0], 101, t)
