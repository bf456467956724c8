"""The tcgen05 GEMM in isolation (through the hs_debug_gemm_bf16 test hook), against plain
fp32 products of the same bf16 operands.  Sizes span several tiles with ragged tails."""
import pytest
import torch

pytestmark = pytest.mark.gpu

hs = pytest.importorskip("paper_2110_08941_gb300")


def _p8(n):
    return (n + 7) // 8 * 8


def _bf(rows, cols, gen):
    """bf16 [rows, pad8(cols)] buffer (padding columns NaN-free random) and its [rows, cols] view."""
    full = torch.randn(rows, _p8(cols), generator=gen, device="cuda").to(torch.bfloat16)
    return full, full[:, :cols]


def _rel(a, b):
    return (torch.linalg.vector_norm((a - b).double()) / torch.linalg.vector_norm(b.double())).item()


SHAPES = [(128, 256, 64), (300, 520, 200), (1, 10, 8), (257, 1000, 1000), (640, 768, 4096), (129, 16, 24),
          (513, 384, 136)]
FORMS = [hs.HS_GEMM_FORM_SINGLE, hs.HS_GEMM_FORM_PAIR]


@pytest.mark.parametrize("form", FORMS)
@pytest.mark.parametrize("M,N,K", SHAPES)
def test_forward_relu(M, N, K, form):
    g = torch.Generator(device="cuda").manual_seed(M * 7 + N)
    A, a = _bf(M, K, g)
    B, b = _bf(N, K, g)
    bias = torch.randn(N, generator=g, device="cuda")
    D = torch.full((M, _p8(N)), float("nan"), dtype=torch.bfloat16, device="cuda")
    hs.hs_debug_gemm_bf16(hs.HS_GEMM_FWD_RELU | form, M, N, K, A, B, D, bias=bias)
    ref = torch.relu(a.float() @ b.float().t() + bias)
    got = D[:, :N].float()
    assert _rel(got, ref) < 6e-3
    assert torch.all(got >= 0)


@pytest.mark.parametrize("form", FORMS)
@pytest.mark.parametrize("M,N,K", SHAPES)
def test_forward_logits(M, N, K, form):
    g = torch.Generator(device="cuda").manual_seed(M + 3 * N + K)
    A, a = _bf(M, K, g)
    B, b = _bf(N, K, g)
    bias = torch.randn(N, generator=g, device="cuda")
    D = torch.full((M, _p8(N)), float("nan"), device="cuda")
    hs.hs_debug_gemm_bf16(hs.HS_GEMM_FWD_LOGITS | form, M, N, K, A, B, D, bias=bias)
    ref = a.float() @ b.float().t() + bias
    assert _rel(D[:, :N], ref) < 1e-5


@pytest.mark.parametrize("form", FORMS)
@pytest.mark.parametrize("M,N,K", SHAPES)
def test_input_gradient_mask(M, N, K, form):
    g = torch.Generator(device="cuda").manual_seed(5 * M + N + 11 * K)
    A, a = _bf(M, K, g)
    B, b = _bf(K, N, g)                     # MN-major operand: [K rows][N]
    Z, z = _bf(M, N, g)
    D = torch.full((M, _p8(N)), float("nan"), dtype=torch.bfloat16, device="cuda")
    hs.hs_debug_gemm_bf16(hs.HS_GEMM_DGRAD | form, M, N, K, A, B, D, Z=Z)
    ref = (a.float() @ b.float()) * (z.float() > 0)
    got = D[:, :N].float()
    assert _rel(got, ref) < 6e-3
    assert torch.all(got[z.float() <= 0] == 0)


@pytest.mark.parametrize("M,N,groups", [(128, 256, [64]), (300, 520, [1, 63, 64, 65, 200]),
                                        (10, 256, [43, 85, 128, 256]), (1000, 512, [242, 2410, 316]),
                                        (256, 768, [7] * 40)])
@pytest.mark.parametrize("form", FORMS)
def test_weight_gradient_grouped(M, N, groups, form):
    g = torch.Generator(device="cuda").manual_seed(M + N + len(groups))
    K = sum(groups)
    ko = [0]
    for n in groups:
        ko.append(ko[-1] + n)
    A, a = _bf(K, M, g)                     # delta rows [K][M] (MN-major)
    B, b = _bf(K, N, g)                     # activations [K][N] (MN-major)
    G = len(groups)
    stride = M * N + 64
    D = torch.full((G * stride,), float("nan"), device="cuda")
    hs.hs_debug_gemm_bf16(hs.HS_GEMM_WGRAD | form, M, N, 0, A, B, D[: M * N].view(M, N), k_offsets=ko, d_gstride=stride)
    for gi in range(G):
        ref = a[ko[gi]:ko[gi + 1]].float().t() @ b[ko[gi]:ko[gi + 1]].float()
        got = D[gi * stride: gi * stride + M * N].view(M, N)
        assert _rel(got, ref) < 1e-5, gi
        assert torch.isnan(D[gi * stride + M * N: (gi + 1) * stride]).all()
