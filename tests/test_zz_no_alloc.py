"""spec_gemm_bf16_noalloc, the split-K projection for callers that cannot allocate device memory
(code under CUDA-graph stream capture, runtimes that hand out memory only from their own fixed
pool): through the C ABI its output matches spec_gemm_bf16 within the GEMM tests' tolerance on
two calls in a row that share the library's fixed scratch; the 128- and 256-row tile variants
with their cross-CTA split-K reduction match the fp64 product; the device guard flag the
kernels would set stays clear (spec_sync(NULL)); and a problem larger than the scratch is
rejected.  Collected last so that a failure here stops a run only after every other test."""
import pytest
import torch

from paper_2609_03181_gb300 import fastmtp as F

pytestmark = pytest.mark.gpu


def _inputs(M, N, K, seed):
    g = torch.Generator().manual_seed(seed)
    X = (torch.randn(M, K, generator=g) * 0.5).to(torch.bfloat16)
    W = (torch.randn(N, K, generator=g) * 0.02).to(torch.bfloat16)
    return X, W


def _splits(N, K):
    """The entry point's documented split rule: min(SM count / weight tiles, K/128, 8)."""
    sms = torch.cuda.get_device_properties(0).multi_processor_count
    return max(1, min(sms // ((N + 127) // 128), (K // 64) // 2, 8))


def test_noalloc_matches_gemm_on_two_calls_in_a_row():
    for call, (M, N, K) in enumerate([(32, 1280, 1280), (8, 3840, 2560)]):
        X, W = _inputs(M, N, K, 100 + call)
        X, W = X.cuda(), W.cuda()
        ref = F.gemm_bf16(X, W)
        Y = torch.full((M, N), float("nan"), dtype=torch.float32, device="cuda")
        F.gemm_bf16_noalloc(X, W, Y)
        torch.cuda.synchronize()
        err = float((Y - ref).abs().max() / ref.abs().max())
        assert err < 1e-4, f"call {call}: relative error {err}"
    F.device_sync()


@pytest.mark.parametrize("M,N,K", [(128, 512, 1280), (256, 256, 1280), (200, 384, 1280), (65, 1024, 896)])
def test_noalloc_large_row_tiles_match_fp64(M, N, K):
    """Row tiles of 128 and 256 (the 256-column kernel variant) and a ragged 65-row case, each
    split several ways along K and reduced across CTAs through the fixed scratch."""
    assert _splits(N, K) > 1
    X, W = _inputs(M, N, K, 7 * M + N)
    ref = X.double() @ W.double().T
    Xd, Wd = X.cuda(), W.cuda()
    Y = torch.full((M, N), float("nan"), dtype=torch.float32, device="cuda")
    F.gemm_bf16_noalloc(Xd, Wd, Y)
    F.device_sync()
    err = float((Y.double().cpu() - ref).abs().max() / ref.abs().max())
    assert err < 1e-4, f"relative error {err}"
    # the unsplit engine sums K in one order, the split one in `splits` partial sums: the two
    # agree to rounding but not bit for bit, which shows the split path ran
    assert not torch.equal(Y, F.gemm_bf16(Xd, Wd))


def test_noalloc_rejects_problems_beyond_its_scratch():
    X, W = _inputs(256, 8192, 1280, 7)
    Y = torch.empty(256, 8192, dtype=torch.float32, device="cuda")
    with pytest.raises(F.FastMTPError) as e:
        F.gemm_bf16_noalloc(X.cuda(), W.cuda(), Y)
    assert e.value.status == F.SPEC_EINVAL and "scratch" in str(e.value)
