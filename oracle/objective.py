"""Plain fp64 oracle of the FastMTP draft-head training objective (Sec. 5.6, "Draft-head
objective", the CE / KL / MSE equations and their weighted sum).

TEST INFRASTRUCTURE: imported only by tests/, __graft_entry__.smoke() and bench.py's
CPU-baseline leg.  Nothing in the product library imports, links or runs it.

For every valid response row p and recursive depth k = 1..K the paper defines the draft
distribution P_p^(k) = softmax(l_p^(k)) with l_p^(k) = W_lm u_p^(k) (the tied LM head applied
to the draft state), the detached verifier distribution Q_p = softmax(W_lm b_{p+1}), and

  CE_k  = E_p[ -log P_p^(k)(x_{p+2}) ]
  KL_k  = E_p[ KL(Q_p || P_p^(k)) ] = E_p[ sum_v Q_p(v) (log Q_p(v) - log P_p^(k)(v)) ]
  MSE_k = E_p[ || u_p^(k) - b_{p+1} ||_2^2 ]

with every depth using the same row-aligned targets x_{p+2} and b_{p+1}.  The expectations
are means over the valid rows (prompt and padding rows excluded).  With
alpha_k = beta^(k-1) / sum_r beta^(r-1) (beta = 0.6) the objective is

  L = 0.85 sum_k alpha_k CE_k + 0.45 sum_k alpha_k KL_k + 0.45 sum_k alpha_k MSE_k.

Everything is fp64 from the bf16-stored inputs (u, b, W_lm); each function follows the
definition above term by term.  Pins: tests/test_objective_pins.py."""
from __future__ import annotations

from dataclasses import dataclass
from typing import List, Optional

import torch

F64 = torch.float64

PAPER_BETA = 0.6
PAPER_WEIGHTS = (0.85, 0.45, 0.45)   # CE, KL, MSE


def depth_weights(K: int, beta: float = PAPER_BETA) -> List[float]:
    """alpha_k = beta^(k-1) / sum_{r=1..K} beta^(r-1), k = 1..K."""
    z = sum(beta ** (r - 1) for r in range(1, K + 1))
    return [beta ** (k - 1) / z for k in range(1, K + 1)]


@dataclass
class DraftLoss:
    total: float
    ce: List[float]          # [K] means over valid rows
    kl: List[float]
    mse: List[float]
    alpha: List[float]
    row_ce: torch.Tensor     # [K][R] per row (invalid rows included, not averaged)
    row_kl: torch.Tensor
    row_mse: torch.Tensor


def draft_loss(u: torch.Tensor, b_next: torch.Tensor, target: torch.Tensor, lm_head: torch.Tensor,
               valid: Optional[torch.Tensor] = None, beta: float = PAPER_BETA,
               weights=PAPER_WEIGHTS) -> DraftLoss:
    """u: [K][R][d] draft states u_p^(k); b_next: [R][d] verifier states b_{p+1}; target: [R]
    token ids x_{p+2}; lm_head: [V][d]; valid: [R] bool (None: every row)."""
    K, R, d = u.shape
    W = lm_head.to(F64)
    b = b_next.to(F64)
    valid = torch.ones(R, dtype=torch.bool) if valid is None else valid.to(torch.bool)
    tgt = target.to(torch.long)
    log_q = torch.log_softmax(b @ W.T, dim=-1)            # log Q_p(v)
    q = torch.exp(log_q)
    row_ce = torch.zeros(K, R, dtype=F64)
    row_kl = torch.zeros(K, R, dtype=F64)
    row_mse = torch.zeros(K, R, dtype=F64)
    for k in range(K):
        uk = u[k].to(F64)
        log_p = torch.log_softmax(uk @ W.T, dim=-1)       # log P_p^(k)(v)
        row_ce[k] = -log_p.gather(1, tgt[:, None])[:, 0]
        row_kl[k] = (q * (log_q - log_p)).sum(-1)
        row_mse[k] = ((uk - b) ** 2).sum(-1)
    n = int(valid.sum())
    mean = lambda x: float(x[valid].sum() / n) if n else 0.0
    ce = [mean(row_ce[k]) for k in range(K)]
    kl = [mean(row_kl[k]) for k in range(K)]
    mse = [mean(row_mse[k]) for k in range(K)]
    alpha = depth_weights(K, beta)
    w_ce, w_kl, w_mse = weights
    total = (w_ce * sum(a * c for a, c in zip(alpha, ce)) + w_kl * sum(a * c for a, c in zip(alpha, kl)) +
             w_mse * sum(a * c for a, c in zip(alpha, mse)))
    return DraftLoss(total, ce, kl, mse, alpha, row_ce, row_kl, row_mse)
