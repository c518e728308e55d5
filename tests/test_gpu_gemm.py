"""Kernel test of the GEMMs: tcgen05 (one pass and split-K), the many-row
kernel (query, GELU and residual epilogues; K split over a cluster pair) and
SIMT against a plain PyTorch fp32 matmul of the same bf16 operands."""
import pytest
import torch

pytestmark = pytest.mark.gpu

SHAPES = [(128, 16, 64), (300, 9, 1280), (3840, 9, 1280), (1280, 40, 5120), (517, 200, 384),
          (1024, 256, 768), (640, 448, 1280), (51866, 9, 1280), (256, 137, 3072), (1280, 544, 3072),
          (3840, 448, 1280)]


@pytest.mark.parametrize("impl", [0, 2, 4, 1])
@pytest.mark.parametrize("M,N,K", SHAPES)
def test_gemm_matches_torch(built_lib, cuda, impl, M, N, K):
    from paper_2608_12703_gb300 import asrspec as A
    g = torch.Generator(device="cpu").manual_seed(M * 7 + N * 3 + K)
    a = torch.randn(M, K, generator=g).to(torch.bfloat16).to(cuda)
    b = torch.randn(N, K, generator=g).to(torch.bfloat16).to(cuda)
    c = torch.full((M, N), float("nan"), device=cuda)
    A.asr_spec_test_gemm(impl, a, b, c, M, N, K, torch.cuda.current_stream().cuda_stream)
    ref = a.float() @ b.float().T
    err = (c - ref).abs().max().item()
    assert err <= 1e-4 * K ** 0.5 * 4, err


@pytest.mark.parametrize("M,N,K", [(51866, 9, 1280), (51865, 448, 384), (1000, 256, 768), (3000, 137, 64)])
def test_fused_argmax_matches_torch(built_lib, cuda, M, N, K):
    """The LM-head epilogue (per-column argmax, no logits stored) over every N tile width."""
    from paper_2608_12703_gb300 import asrspec as A
    g = torch.Generator(device="cpu").manual_seed(M + N + K)
    a = torch.randn(M, K, generator=g).to(torch.bfloat16).to(cuda)
    b = torch.randn(N, K, generator=g).to(torch.bfloat16).to(cuda)
    c = torch.full((N,), -1.0, device=cuda)
    A.asr_spec_test_gemm(3, a, b, c, M, N, K, torch.cuda.current_stream().cuda_stream)
    ref = a.float() @ b.float().T
    got = c.long()
    best = ref.max(dim=0).values
    # exact unless two columns entries tie within fp32 summation-order noise
    picked = ref[got, torch.arange(N, device=cuda)]
    assert torch.all(best - picked <= 1e-3 * K ** 0.5), (best - picked).max()
    assert (got == ref.argmax(dim=0)).float().mean() > 0.99


WIDE_SHAPES = [(1280, 448, 1280), (3840, 448, 1280), (5120, 448, 1280), (1280, 448, 5120), (768, 144, 3072),
               (2304, 544, 768), (256, 65, 64), (128, 300, 128)]


@pytest.mark.parametrize("impl", [5, 6, 7])
@pytest.mark.parametrize("M,N,K", WIDE_SHAPES)
def test_wide_gemm_matches_torch(built_lib, cuda, impl, M, N, K):
    """The many-row kernel's tile choices (N tiles of 32 .. 160, ragged last
    tile, K split in two from 48 k-blocks); GELU against torch's erf GELU
    within the bf16 rounding of the stored result."""
    from paper_2608_12703_gb300 import asrspec as A
    g = torch.Generator(device="cpu").manual_seed(M * 5 + N + K * 3)
    a = (0.25 * torch.randn(M, K, generator=g)).to(torch.bfloat16).to(cuda)
    b = torch.randn(N, K, generator=g).to(torch.bfloat16).to(cuda)
    c = torch.full((N, M), float("nan"), device=cuda)
    A.asr_spec_test_gemm(impl, a, b, c, M, N, K, torch.cuda.current_stream().cuda_stream)
    ref = (a.float() @ b.float().T).T
    if impl == 6:
        ref = torch.nn.functional.gelu(ref)
        err = ((c - ref).abs() - 8e-3 * ref.abs()).max().item()
        assert err <= 1e-4 * K ** 0.5, err
    else:
        err = (c - ref).abs().max().item()
        assert err <= 1e-4 * K ** 0.5, err
