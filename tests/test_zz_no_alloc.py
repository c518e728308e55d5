"""The allocation-free split-K GEMM entry point against the allocating one.

Callers that may not allocate device memory (a framework owning the device
pool, a serving loop that forbids allocation after start-up, code running
during another thread's graph capture) use asr_spec_gemm_noalloc, whose
scratch is one fixed device array shared by every call.  Two calls in a row
with different data must each match asr_spec_test_gemm (split-K with its own
workspace) within the GEMM tests' tolerance, so nothing left in the shared
array from one call leaks into the next.  The file sorts last so that a run
stopping at its first failure has run every other test before it.
"""
import pytest

pytestmark = pytest.mark.gpu


def test_noalloc_gemm_matches_allocating_entry_two_calls(built_lib, cuda):
    import torch
    from paper_2608_12703_gb300 import asrspec as A
    st = torch.cuda.current_stream().cuda_stream
    for call, (M, N, K) in enumerate([(3840, 9, 1280), (1280, 137, 5120)]):
        g = torch.Generator(device="cpu").manual_seed(100 + call)
        a = torch.randn(M, K, generator=g).to(torch.bfloat16).to(cuda)
        b = torch.randn(N, K, generator=g).to(torch.bfloat16).to(cuda)
        ref = torch.full((M, N), float("nan"), device=cuda)
        out = torch.full((M, N), float("nan"), device=cuda)
        A.asr_spec_test_gemm(2, a, b, ref, M, N, K, st)          # 3-way split, allocated workspace
        torch.cuda.synchronize()
        A.asr_spec_gemm_noalloc(a, b, out, M, N, K, 3, st)
        torch.cuda.synchronize()
        tol = 1e-4 * K ** 0.5 * 4
        assert torch.isfinite(out).all()
        assert (out - ref).abs().max().item() <= tol
        assert (out - a.float() @ b.float().T).abs().max().item() <= tol


def test_noalloc_gemm_rejects_oversize(built_lib, cuda):
    import torch
    from paper_2608_12703_gb300 import asrspec as A
    a = torch.zeros(51866, 1280, dtype=torch.bfloat16, device=cuda)
    b = torch.zeros(256, 1280, dtype=torch.bfloat16, device=cuda)
    c = torch.zeros(51866, 256, device=cuda)
    with pytest.raises(A.AsrSpecError, match="ASR_E_CAPACITY"):
        A.asr_spec_gemm_noalloc(a, b, c, 51866, 256, 1280, 20, torch.cuda.current_stream().cuda_stream)
