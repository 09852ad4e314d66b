"""spec_draft_loss through the C ABI against the fp64 oracle of the draft-head objective
(Sec. 5.6, CE / KL / MSE per depth and their alpha-weighted sum), on the same bf16 inputs.

Rules: per-row and mean CE and MSE within relative 1e-4, KL within 1e-4 absolute + 1e-3
relative (it is a difference of log-sum-exps; the GPU sums the logits in fp32), the weighted
total within relative 1e-4.  Cases: a ragged last vocabulary tile, every row-group size (K = 1,
2, 3, 5), the full 129,280-token vocabulary with one and with two 256-row activation tiles,
logits ten times larger (the softmax statistics must stay stable), masked rows and an
out-of-range target."""
import math

import numpy as np
import pytest
import torch

import oracle as O
import synth_inputs as S
from paper_2609_03181_gb300 import fastmtp as F

pytestmark = pytest.mark.gpu

D = 1280


def make_case(K, R, V, seed, state_std=1.0, w_std=0.02, invalid_every=0):
    u = S.normal(seed, "obj.u", (K, R, D), state_std)
    b = S.normal(seed, "obj.b", (R, D), state_std)
    W = S.normal(seed, "obj.w", (V, D), w_std)
    tgt = torch.from_numpy(S.integers(seed, "obj.t", R, 0, V - 1).astype(np.int32))
    valid = torch.ones(R, dtype=torch.int32)
    if invalid_every:
        valid[::invalid_every] = 0
    return u, b, W, tgt, valid


def check(K, R, V, seed, **kw):
    u, b, W, tgt, valid = make_case(K, R, V, seed, **kw)
    ref = O.draft_loss(u, b, tgt, W, valid=valid.bool())
    out, rows = F.draft_loss(u.cuda(), b.cuda(), tgt.cuda(), W.cuda(), valid=valid.cuda())
    torch.cuda.synchronize()
    out, rows = out.double().cpu(), rows.double().cpu()
    for k in range(K):
        assert torch.allclose(rows[k, :, 0], ref.row_ce[k], rtol=1e-4, atol=0), (k, "ce")
        assert torch.allclose(rows[k, :, 1], ref.row_kl[k], rtol=1e-3, atol=1e-4), (k, "kl")
        assert torch.allclose(rows[k, :, 2], ref.row_mse[k], rtol=1e-4, atol=0), (k, "mse")
        assert abs(out[1 + k] - ref.ce[k]) <= 1e-4 * abs(ref.ce[k])
        assert abs(out[1 + K + k] - ref.kl[k]) <= 1e-4 + 1e-3 * abs(ref.kl[k])
        assert abs(out[1 + 2 * K + k] - ref.mse[k]) <= 1e-4 * abs(ref.mse[k])
    assert abs(out[0] - ref.total) <= 1e-4 * abs(ref.total)
    F.device_sync()
    return out, ref


@pytest.mark.parametrize("K,R,V", [(3, 20, 5000), (1, 7, 1000), (2, 33, 4100), (5, 9, 2048)])
def test_objective_matches_oracle_small_vocab(K, R, V):
    check(K, R, V, seed=K * 100 + R, invalid_every=4)


def test_objective_full_vocab_one_and_two_row_tiles():
    check(3, 64, 129280, seed=7)                       # 256 packed rows: one 256-row tile
    check(3, 100, 129280, seed=8, invalid_every=3)     # 400 packed rows: two tiles


def test_objective_large_logits_stay_stable():
    # logits ~ N(0, 7^2): exp() of the raw values would overflow fp32 without the running maxima
    out, ref = check(3, 16, 20000, seed=9, w_std=0.2)
    assert all(math.isfinite(x) for x in out.tolist())


def test_objective_bad_target_gives_nan_row():
    u, b, W, tgt, valid = make_case(2, 5, 3000, seed=10)
    tgt[3] = 3000
    out, rows = F.draft_loss(u.cuda(), b.cuda(), tgt.cuda(), W.cuda())
    torch.cuda.synchronize()
    assert torch.isnan(rows[:, 3, 0]).all() and not torch.isnan(rows[:, [0, 1, 2, 4], 0]).any()


def test_objective_rejects_a_small_workspace():
    u, b, W, tgt, valid = make_case(3, 8, 1000, seed=11)
    ws = torch.empty(1024, dtype=torch.uint8, device="cuda")
    with pytest.raises(F.FastMTPError) as e:
        F.draft_loss(u.cuda(), b.cuda(), tgt.cuda(), W.cuda(), workspace=ws)
    assert e.value.status == F.SPEC_EINVAL and "workspace" in str(e.value)
