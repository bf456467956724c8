"""Device-side failure detection without a GPU fault: a product whose TMA producer issues no
loads (the test hook's stall flag) lets the tensor-core kernel's bounded waits expire; the kernel
records the expiry in its status word, raises its abort flag, frees its tensor memory and returns,
the call reports HS_ERR_DEVICE_CHECK within seconds, and the device stays usable."""
import time

import pytest
import torch

import paper_2110_08941_gb300 as hs

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("form", [hs.HS_GEMM_FORM_SINGLE, hs.HS_GEMM_FORM_PAIR])
def test_expired_wait_is_reported_and_the_device_stays_usable(form):
    g = torch.Generator(device="cuda").manual_seed(3)
    M, N, K = 300, 520, 200
    A = torch.randn(M, K, generator=g, device="cuda").to(torch.bfloat16)
    B = torch.randn(N, K, generator=g, device="cuda").to(torch.bfloat16)
    bias = torch.randn(N, generator=g, device="cuda")
    D = torch.full((M, N), float("nan"), device="cuda")
    t0 = time.perf_counter()
    with pytest.raises(hs.HsError) as e:
        hs.hs_debug_gemm_bf16(hs.HS_GEMM_FWD_LOGITS | form | hs.HS_GEMM_TEST_STALL, M, N, K, A, B, D, bias=bias)
    assert e.value.status == hs.HS_ERR_DEVICE_CHECK
    assert time.perf_counter() - t0 < 30.0          # bounded: a 2 s limit per wait
    torch.cuda.synchronize()
    hs.hs_debug_gemm_bf16(hs.HS_GEMM_FWD_LOGITS | form, M, N, K, A, B, D, bias=bias)
    ref = A.float() @ B.float().t() + bias
    assert torch.allclose(D, ref, rtol=1e-4, atol=1e-3)
