"""Pins of the fp64 oracle of the draft-head objective (Sec. 5.6, CE / KL / MSE and their
alpha-weighted sum) against hand-worked numbers, closed forms and library routines (CPU)."""
import math

import numpy as np
import pytest
import torch
import torch.nn.functional as F

import oracle as O

F64 = torch.float64


def test_depth_weights_hand_values():
    # beta = 0.6, K = 3: (1, 0.6, 0.36) / 1.96
    a = O.depth_weights(3)
    assert all(abs(x - y) < 1e-15 for x, y in zip(a, [1 / 1.96, 0.6 / 1.96, 0.36 / 1.96]))
    assert O.depth_weights(1) == [1.0]
    assert abs(sum(O.depth_weights(5, 0.3)) - 1.0) < 1e-15


def test_hand_worked_three_token_example():
    """V = 3, d = 2, W_lm = [[1,0],[0,1],[0,0]]: b = (ln 2, 0) gives Q = (1/2, 1/4, 1/4);
    u = (0, ln 3) gives P = (1/5, 3/5, 1/5).  Target token 1."""
    W = torch.tensor([[1.0, 0.0], [0.0, 1.0], [0.0, 0.0]], dtype=F64)
    b = torch.tensor([[math.log(2.0), 0.0]], dtype=F64)
    u = torch.tensor([[[0.0, math.log(3.0)]]], dtype=F64)
    r = O.draft_loss(u, b, torch.tensor([1]), W)
    ce = math.log(5.0 / 3.0)
    kl = 0.5 * math.log(0.5 / 0.2) + 0.25 * math.log(0.25 / 0.6) + 0.25 * math.log(0.25 / 0.2)
    mse = math.log(2.0) ** 2 + math.log(3.0) ** 2
    assert abs(r.ce[0] - ce) < 1e-14 and abs(r.kl[0] - kl) < 1e-14 and abs(r.mse[0] - mse) < 1e-14
    assert abs(r.total - (0.85 * ce + 0.45 * kl + 0.45 * mse)) < 1e-14


def test_uniform_logits_and_identical_states():
    g = torch.Generator().manual_seed(1)
    V, d, R, K = 50, 8, 6, 3
    b = torch.randn(R, d, generator=g, dtype=F64)
    u = b.expand(K, R, d).clone()
    tgt = torch.randint(0, V, (R,), generator=g)
    # W_lm = 0: every distribution is uniform, CE = log V, KL = 0; u = b: MSE = 0
    r = O.draft_loss(u, b, tgt, torch.zeros(V, d, dtype=F64))
    assert all(abs(c - math.log(V)) < 1e-12 for c in r.ce)
    assert all(abs(x) < 1e-12 for x in r.kl) and all(x == 0.0 for x in r.mse)
    # any W_lm: identical draft and verifier states make P = Q, so KL = 0 at every depth
    W = torch.randn(V, d, generator=g, dtype=F64)
    r = O.draft_loss(u, b, tgt, W)
    assert all(abs(x) < 1e-12 for x in r.kl)
    assert abs(r.ce[0] - r.ce[2]) < 1e-12


def test_terms_match_library_routines_and_mask():
    g = torch.Generator().manual_seed(2)
    V, d, R, K = 97, 16, 9, 2
    W = torch.randn(V, d, generator=g, dtype=F64) * 0.5
    b = torch.randn(R, d, generator=g, dtype=F64)
    u = torch.randn(K, R, d, generator=g, dtype=F64)
    tgt = torch.randint(0, V, (R,), generator=g)
    valid = torch.tensor([1, 1, 0, 1, 0, 1, 1, 1, 0], dtype=torch.bool)
    r = O.draft_loss(u, b, tgt, W, valid=valid)
    lq = F.log_softmax(b @ W.T, -1)
    for k in range(K):
        lp = F.log_softmax(u[k] @ W.T, -1)
        ce_rows = F.cross_entropy(u[k] @ W.T, tgt, reduction="none")
        kl_rows = F.kl_div(lp, lq, log_target=True, reduction="none").sum(-1)   # KL(Q || P)
        assert torch.allclose(r.row_ce[k], ce_rows, atol=1e-12)
        assert torch.allclose(r.row_kl[k], kl_rows, atol=1e-12)
        for row in range(R):   # Gibbs: KL >= 0, and scipy's relative entropy agrees
            Q = torch.exp(lq[row]).numpy()
            P = torch.exp(lp[row]).numpy()
            assert r.row_kl[k, row] >= 0
            assert abs(float(np.sum(Q * np.log(Q / P))) - float(r.row_kl[k, row])) < 1e-10
        assert abs(r.ce[k] - float(ce_rows[valid].mean())) < 1e-12
        assert abs(r.mse[k] - float(((u[k] - b) ** 2).sum(-1)[valid].mean())) < 1e-12
    a = [1 / 1.6, 0.6 / 1.6]
    hand = (0.85 * (a[0] * r.ce[0] + a[1] * r.ce[1]) + 0.45 * (a[0] * r.kl[0] + a[1] * r.kl[1]) +
            0.45 * (a[0] * r.mse[0] + a[1] * r.mse[1]))
    assert abs(r.total - hand) < 1e-12
    # the excluded rows change nothing
    tgt2 = tgt.clone()
    tgt2[~valid] = 0
    u2 = u.clone()
    u2[:, ~valid] = 7.0
    r2 = O.draft_loss(u2, b, tgt2, W, valid=valid)
    assert abs(r2.total - r.total) < 1e-12
