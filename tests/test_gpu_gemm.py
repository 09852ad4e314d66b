"""The tcgen05 GEMM engine (spec_gemm_bf16) against the fp64 product of the same bf16 inputs,
over several tiles, ragged row and column tails and every activation box height."""
import pytest
import torch

from paper_2609_03181_gb300 import fastmtp as F

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("M,N,K", [(1, 128, 64), (5, 300, 1280), (16, 1280, 896), (33, 1280, 1280),
                                   (64, 3840, 1280), (100, 640, 2560), (256, 384, 128), (300, 256, 3584),
                                   (1000, 129, 192)])
def test_gemm_matches_fp64_product(M, N, K):
    g = torch.Generator().manual_seed(M * 7 + N + K)
    X = (torch.randn(M, K, generator=g) * 0.5).to(torch.bfloat16)
    W = (torch.randn(N, K, generator=g) * 0.02).to(torch.bfloat16)
    Y = F.gemm_bf16(X.cuda(), W.cuda())
    torch.cuda.synchronize()
    ref = X.double() @ W.double().T
    err = (Y.double().cpu() - ref).abs().max() / ref.abs().max()
    assert err < 1e-4, f"relative error {err}"   # fp32 accumulation of exact bf16 products


def test_gemm_rows_do_not_depend_on_batch():
    """A row's result is bit-identical whether it is computed alone or with 200 other rows."""
    g = torch.Generator().manual_seed(1)
    X = (torch.randn(201, 1280, generator=g)).to(torch.bfloat16).cuda()
    W = (torch.randn(1280, 1280, generator=g) * 0.02).to(torch.bfloat16).cuda()
    full = F.gemm_bf16(X, W)
    for i in (0, 17, 200):
        one = F.gemm_bf16(X[i:i + 1].contiguous(), W)
        assert torch.equal(one[0], full[i])


@pytest.mark.parametrize("M,N,K", [(16, 256, 128), (16, 256, 1280), (64, 384, 4096), (200, 128, 896)])
def test_gemm_e4m3_matches_fp64_product(M, N, K):
    """spec_gemm_e4m3 (tcgen05 kind::f8f6f4) against the fp64 product of the decoded codes times
    the row scales.  Codes of N(0, 1) values (no NaN codes)."""
    import oracle as O
    g = torch.Generator().manual_seed(M + N + K)
    X8 = (torch.randn(M, K, generator=g) * 2).clamp(-448, 448).to(torch.float8_e4m3fn).view(torch.uint8)
    W8 = torch.randn(N, K, generator=g).clamp(-448, 448).to(torch.float8_e4m3fn).view(torch.uint8)
    sc = torch.rand(N, generator=g) + 0.5
    Y = F.gemm_e4m3(X8.cuda(), W8.cuda(), sc.cuda())
    F.device_sync()
    ref = (O.decode_e4m3(X8) @ O.decode_e4m3(W8).T) * sc.double()
    err = float((Y.double().cpu() - ref).abs().max() / ref.abs().max())
    print(f"[e4m3 gemm] M={M} N={N} K={K}: relative error {err:.3g}")
    assert err < 1e-4, f"relative error {err}"
