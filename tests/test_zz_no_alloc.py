"""spec_gemm_bf16_noalloc, the split-K projection for callers that cannot allocate device memory
(stream capture, fixed-pool runtimes): through the C ABI its output matches spec_gemm_bf16 within
the GEMM tests' tolerance, on two calls in a row that share the library's fixed scratch, and it
rejects a problem larger than that scratch.  Collected last so that a failure here stops a run
only after every other test."""
import pytest
import torch

from paper_2609_03181_gb300 import fastmtp as F

pytestmark = pytest.mark.gpu


def _inputs(M, N, K, seed):
    g = torch.Generator().manual_seed(seed)
    X = (torch.randn(M, K, generator=g) * 0.5).to(torch.bfloat16).cuda()
    W = (torch.randn(N, K, generator=g) * 0.02).to(torch.bfloat16).cuda()
    return X, W


def test_noalloc_matches_gemm_on_two_calls_in_a_row():
    for call, (M, N, K) in enumerate([(32, 1280, 1280), (8, 3840, 2560)]):
        X, W = _inputs(M, N, K, 100 + call)
        ref = F.gemm_bf16(X, W)
        Y = torch.full((M, N), float("nan"), dtype=torch.float32, device="cuda")
        F.gemm_bf16_noalloc(X, W, Y)
        torch.cuda.synchronize()
        err = float((Y - ref).abs().max() / ref.abs().max())
        assert err < 1e-4, f"call {call}: relative error {err}"


def test_noalloc_rejects_problems_beyond_its_scratch():
    X, W = _inputs(256, 8192, 1280, 7)
    Y = torch.empty(256, 8192, dtype=torch.float32, device="cuda")
    with pytest.raises(F.FastMTPError) as e:
        F.gemm_bf16_noalloc(X, W, Y)
    assert e.value.status == F.SPEC_EINVAL and "scratch" in str(e.value)
