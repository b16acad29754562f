"""The Newton-Schulz product of Gefen-Muon (gefen_gemm_bf16: C = alpha A B^T +
beta D, bf16 storage, fp32 accumulation) against PyTorch's fp32 product of
the same bf16 operands, rounded once to bf16.  Summation order differs, so an
element may round to the neighbouring bf16 value: within 2^-7 relative plus
2^-12 of the largest |C|.  Shapes: one tile, several tiles and k-tiles (the
operand ring wraps), ragged M, N and K, the Newton-Schulz shapes of a
2048 x 8192 matrix, the transposed output, and leading dimensions that TMA
cannot address (the CUDA-core path: lda = 100, and ldc = 700 in the 300 x 700
case).  A last wave of tiles that fills at most half the SMs runs as half
tiles: 2048 x 8192 and 2904 x 4008 (256-wide tiles), 2048 x 1536 (128-wide)."""
import pytest
import torch

from paper_2606_13894_gb300 import gefen as G

pytestmark = pytest.mark.gpu


def _ref(A, B, alpha, beta, D):
    r = alpha * (A.float() @ B.float().T)
    if beta != 0.0:
        r = r + beta * D.float()
    return r


def _close(got, ref):
    tol = 2.0 ** -7 * ref.abs() + 2.0 ** -12 * ref.abs().max()
    bad = (got.float() - ref).abs() > tol
    assert not bool(bad.any()), f"{int(bad.sum())} of {bad.numel()} outside; max err {float((got.float() - ref).abs().max())}"


@pytest.mark.parametrize("M,N,K", [(128, 256, 64), (256, 512, 1024), (296, 712, 200), (64, 64, 256),
                                   (2048, 2048, 8192), (2048, 8192, 2048), (96, 512, 96),
                                   (2904, 4008, 328), (300, 700, 200), (2048, 1536, 256)])
@pytest.mark.parametrize("with_d", [False, True])
def test_gemm_matches_fp32_product(M, N, K, with_d):
    g = torch.Generator(device="cuda").manual_seed(M * 7 + N + K)
    A = torch.randn(M, K, device="cuda", generator=g).to(torch.bfloat16)
    B = torch.randn(N, K, device="cuda", generator=g).to(torch.bfloat16)
    D = torch.randn(M, N, device="cuda", generator=g).to(torch.bfloat16) if with_d else None
    alpha, beta = (-4.775, 2.0315) if with_d else (1.0, 0.0)
    C = torch.empty(M, N, dtype=torch.bfloat16, device="cuda")
    CT = torch.empty(N, M, dtype=torch.bfloat16, device="cuda")
    _, _, ws = G.gefen_gemm_bf16(A, B, alpha=alpha, beta=beta, D=D, C=C, CT=CT)
    G.gefen_step_status(ws)  # no bounded wait gave up
    ref = _ref(A, B, alpha, beta, D)
    _close(C, ref)
    assert torch.equal(CT, C.T)


def test_gemm_cuda_core_path_for_unaligned_leading_dimensions():
    g = torch.Generator(device="cuda").manual_seed(5)
    A = torch.randn(70, 100, device="cuda", generator=g).to(torch.bfloat16)   # lda = 100: not a multiple of 8
    B = torch.randn(130, 100, device="cuda", generator=g).to(torch.bfloat16)
    C, _, _ = G.gefen_gemm_bf16(A, B)
    _close(C, _ref(A, B, 1.0, 0.0, None))


def test_gemm_submatrix_operands():
    # leading dimensions larger than the logical widths
    g = torch.Generator(device="cuda").manual_seed(6)
    Abig = torch.randn(256, 640, device="cuda", generator=g).to(torch.bfloat16)
    Bbig = torch.randn(384, 640, device="cuda", generator=g).to(torch.bfloat16)
    A, B = Abig[:, :512], Bbig[:, :512]
    C, _, _ = G.gefen_gemm_bf16(A, B)
    _close(C, _ref(A, B, 1.0, 0.0, None))


@pytest.mark.parametrize("N,K", [(128, 64), (256, 1024), (296, 200), (1000, 96), (2048, 8192), (2048, 2048),
                                 (100, 100)])
@pytest.mark.parametrize("with_d", [False, True])
def test_symmetric_product_is_exactly_symmetric(N, K, with_d):
    # the Newton-Schulz products X X^T and c A A^T + b A: tiles on and above
    # the diagonal, mirrored (N = 100: lda not a multiple of 8, CUDA cores)
    g = torch.Generator(device="cuda").manual_seed(N * 3 + K)
    A = torch.randn(N, K, device="cuda", generator=g).to(torch.bfloat16)
    D = None
    if with_d:
        R = torch.randn(N, N, device="cuda", generator=g)
        D = ((R + R.T) * 0.5).to(torch.bfloat16)
    alpha, beta = (-4.775, 2.0315) if with_d else (1.0, 0.0)
    C, ws = G.gefen_gemm_bf16_sym(A, alpha=alpha, beta=beta, D=D)
    G.gefen_step_status(ws)
    assert torch.equal(C, C.T)
    _close(C, _ref(A, A, alpha, beta, D))
