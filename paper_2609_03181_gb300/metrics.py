"""Speculative-decoding statistics with the definitions of the paper's efficiency table
(Sec. 6.4, Table "Decoding efficiency ... with FastMTP"):

* tau: mean number of tokens committed per speculative step, bonus token included;
* acceptance rate: the position-averaged (tau - 1) / k;
* a_d: probability that draft depth d is accepted given that all shallower depths were;
* c = tau / S: cost of one speculative step in units of one autoregressive step;
* the fixed per-step overhead implied by c: t_AR * (c - 1);
* S = throughput at depth k over greedy decoding (k = 0) of the same setting, and the depth
  that maximises it (the paper's k trade-off: tau grows with k, and so does c).
"""
from __future__ import annotations

import json
import math
from typing import Dict, Iterable, Sequence, Tuple


def tau_from_conditional(a: Sequence[float]) -> float:
    """tau = 1 + a_1 + a_1 a_2 + ... (depth d is reached only if depths < d were accepted)."""
    tau, run = 1.0, 1.0
    for ad in a:
        run *= ad
        tau += run
    return tau


def acceptance_rate(tau: float, k: int) -> float:
    return (tau - 1.0) / k


def step_cost(tau: float, speedup: float) -> float:
    return tau / speedup


def speedup_vs_ar(tok_s: float, ar_tok_s: float, tau: float) -> Dict[str, float]:
    """S = tok_s / ar_tok_s (committed tokens per second at depth k over greedy decoding of the
    same batch and context) and the step cost c = tau / S it implies."""
    S = tok_s / ar_tok_s
    return {"S": S, "c": step_cost(tau, S)}


def best_depth(tok_s_by_k: Dict[int, float]) -> Dict[str, float]:
    """The draft depth with the highest throughput among the measured ones (k = 0 is greedy
    decoding and must be present), and its speedup S over k = 0.  Ties go to the smaller depth."""
    ar = tok_s_by_k[0]
    k = min(tok_s_by_k, key=lambda d: (-tok_s_by_k[d], d))
    return {"k": k, "S": tok_s_by_k[k] / ar}


class DepthPolicy:
    """Draft depth by batch size and context length, from measured throughputs: for every
    measured (batch, context) the depth with the highest committed tokens/s (best_depth); a
    query takes the nearest measured point, by log2 distance in batch first, then in context.
    Built from the JSON lines of `bench.py --sweep` (one router mode) or from a table
    {(batch, ctx): {K: tok_s}} that includes K = 0."""

    def __init__(self, table: Dict[Tuple[int, int], Dict[int, float]]):
        self.best = {key: best_depth(by_k)["k"] for key, by_k in table.items() if 0 in by_k}
        if not self.best:
            raise ValueError("no measured point has the greedy (K = 0) baseline")

    @classmethod
    def from_sweep_lines(cls, lines: Iterable[str], router: str = "uniform") -> "DepthPolicy":
        table: Dict[Tuple[int, int], Dict[int, float]] = {}
        for line in lines:
            line = line.strip()
            if not line:
                continue
            d = json.loads(line)
            if not d.get("sweep") or d.get("router") != router:
                continue
            table.setdefault((int(d["batch"]), int(d["ctx"])), {})[int(d["K"])] = float(d["tokens_per_s"])
        return cls(table)

    @classmethod
    def from_table(cls, table: dict) -> "DepthPolicy":
        """From the packaged table format (depth_table.py): {"points": [{"batch": b, "ctx": c,
        "tokens_per_s": {"0": t0, "1": t1, ...}}, ...]}."""
        t = {(int(p["batch"]), int(p["ctx"])): {int(k): float(v) for k, v in p["tokens_per_s"].items()}
             for p in table["points"]}
        return cls(t)

    def choose(self, batch: int, ctx: int) -> int:
        def dist(key):
            b, c = key
            return (abs(math.log2(b) - math.log2(max(1, batch))), abs(math.log2(c) - math.log2(max(1, ctx))), b, c)
        return self.best[min(self.best, key=dist)]


def fixed_overhead(t_ar: float, c: float) -> float:
    """Extra time of one speculative step over one autoregressive step."""
    return t_ar * (c - 1.0)


def from_accept_hist(hist: Sequence[int]) -> Dict[str, object]:
    """Statistics from a histogram of accepted draft lengths m = 0..K (one entry per verified
    sequence-step).  Committed tokens per step are m + 1."""
    K = len(hist) - 1
    n = sum(hist)
    if n == 0:
        return {"steps": 0, "tau": 0.0, "acceptance_rate": 0.0, "a_d": [0.0] * K}
    tau = sum((m + 1) * c for m, c in enumerate(hist)) / n
    a_d = []
    for d in range(1, K + 1):
        reached = sum(hist[d - 1:])          # depths < d all accepted: m >= d-1
        acc = sum(hist[d:])                  # depth d accepted: m >= d
        a_d.append(acc / reached if reached else 0.0)
    return {"steps": n, "tau": tau, "acceptance_rate": acceptance_rate(tau, K) if K else 0.0, "a_d": a_d}
