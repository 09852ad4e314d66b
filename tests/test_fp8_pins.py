"""Pins of the oracle's fp8 (e4m3) arithmetic of the fp8-expert variant (CPU): rounding to the
nearest e4m3 value against hand-worked numbers (ties to even, the subnormal grid, saturation)
and against PyTorch's float8_e4m3fn conversion, decoding of every byte code against PyTorch's
float8 view, and the per-output-row scales of the dequantised expert matrices."""
import numpy as np
import pytest
import torch

import oracle as O
import synth_inputs as S

F64 = torch.float64


def test_round_e4m3_hand_values():
    x = torch.tensor([1.0625,                 # halfway 1 .. 1.125: even mantissa -> 1
                      1.0625 + 2.0 ** -20,    # just above the tie -> 1.125
                      1.1875,                 # halfway 1.125 .. 1.25: even -> 1.25
                      3.3, -3.3,              # -> 3.25 (step 0.25 in [2, 4))
                      448.0, 460.0, 1.0e4,    # the largest value, rounding to it, saturation
                      2.0 ** -6,              # smallest normal
                      2.0 ** -9, 2.0 ** -10,  # smallest subnormal; half of it ties to 0
                      3 * 2.0 ** -10,         # 1.5 subnormal steps: tie -> 2 steps
                      0.0], dtype=F64)
    want = [1.0, 1.125, 1.25, 3.25, -3.25, 448.0, 448.0, 448.0, 2.0 ** -6, 2.0 ** -9, 0.0, 2.0 ** -8, 0.0]
    assert O.round_e4m3(x).tolist() == want


def test_round_e4m3_matches_library_conversion():
    g = torch.Generator().manual_seed(5)
    x = torch.cat([torch.randn(100000, generator=g, dtype=F64) * s for s in (1e-3, 0.05, 1.0, 30.0, 200.0)])
    x = x.clamp(-448.0, 448.0)
    ref = x.to(torch.float8_e4m3fn).to(F64)
    assert torch.equal(O.round_e4m3(x), ref)


def test_decode_e4m3_every_code():
    codes = torch.arange(256, dtype=torch.int64).to(torch.uint8)
    ref = codes.view(torch.float8_e4m3fn).to(F64)
    got = O.decode_e4m3(codes)
    finite = ~torch.isnan(ref)
    assert int((~finite).sum()) == 2                      # 0x7f and 0xff are NaN in e4m3fn
    assert torch.equal(got[finite], ref[finite])
    # rounding a decoded value gives it back (a fixed point of the grid)
    assert torch.equal(O.round_e4m3(got[finite]), got[finite])


def test_dequant_rows_and_the_quantised_expert_weights():
    sh = S.ModelShape(n_layers=1, n_experts=3, hidden=64, expert_inter=32, vocab=50, n_heads=2, head_dim=32)
    vw = S.verifier_weights(sh, 2)
    v8 = S.quantize_experts_fp8(vw)
    lw = v8.layers[0]
    w = lw.w_gate_up.to(F64)
    deq = O.dequant_rows(lw.w_gate_up_f8, lw.gate_up_scale)
    # every row's largest entry maps to +-448 times its scale, and every entry is within half an
    # e4m3 step (2^-4 relative for normal values) of the bf16 weight
    assert torch.allclose(deq.abs().amax(-1), w.abs().amax(-1), rtol=2 ** -4)
    assert ((deq - w).abs() <= w.abs() * 2.0 ** -4 + lw.gate_up_scale.to(F64)[..., None] * 2.0 ** -9).all()
    # one scale per output row: doubling the scale of down row 5 of expert 1 doubles exactly
    # output feature 5 of that expert's SwiGLU and nothing else
    x = torch.randn(4, sh.hidden, generator=torch.Generator().manual_seed(3), dtype=F64)
    wgu = O.dequant_rows(lw.w_gate_up_f8[1], lw.gate_up_scale[1])
    y0 = O.swiglu(x, wgu, O.dequant_rows(lw.w_down_f8[1], lw.down_scale[1]), rb=True, fp8=True)
    sc = lw.down_scale[1].clone()
    sc[5] *= 2
    y1 = O.swiglu(x, wgu, O.dequant_rows(lw.w_down_f8[1], sc), rb=True, fp8=True)
    assert torch.equal(y1[:, 5], 2 * y0[:, 5])
    keep = [i for i in range(sh.hidden) if i != 5]
    assert torch.equal(y1[:, keep], y0[:, keep])
