"""The 12-layer speculative loop on the GPU against the fp64 oracle's plain greedy decoding: a
16-token slice of the end-to-end workload (the full decoder, vocabulary 129,280, acceptance-
tuned successor-map weights, the FastMTP draft head at K=3) for two sequences.

The committed stream of speculative decoding must equal greedy decoding (Sec. 3.1).  Here the
GPU's speculative stream is compared token by token with the oracle's greedy stream: token i of
a sequence is compared while the oracle's top-1 minus top-2 logit margin at that position
exceeds 8 standard deviations of the logit noise the measured state difference implies (at
least 1e-3), and the comparison of a sequence ends at its first token below that margin (later
tokens depend on it).  At least 16 tokens must be compared."""
import numpy as np
import pytest
import torch

import oracle as O
import synth_inputs as S
from paper_2609_03181_gb300 import fastmtp as F
from tests.gpu_util import argmax_margin, rel_err, REL_TOL

pytestmark = pytest.mark.gpu

B, K, N_TOK, SEED = 2, 3, 16, 3


def test_speculative_stream_matches_oracle_greedy_12_layers():
    shape = S.ModelShape()
    vw, dw, _ = S.successor_weights(shape, SEED, 7.0)
    ctx = [int(c) for c in S.integers(SEED, "ctx.slice", B, 300, 600)]
    kvs = [S.kv_prefix(SEED, b, shape.n_layers, ctx[b], shape.n_heads, shape.head_dim) for b in range(B)]
    dkvs = [S.draft_kv_prefix(SEED, b, ctx[b], shape.n_heads, shape.head_dim) for b in range(B)]
    pend = [int(t) for t in S.integers(SEED, "pending.slice", B, 0, shape.vocab - 1)]

    # ---- GPU: one K=0 step (the first base state), then speculative steps of the draft head
    eng = F.Engine(vw, dw, max_batch=B, K_max=K, max_ctx=max(ctx) + N_TOK + 2 * (K + 1) + 8, page_size=64)
    for b in range(B):
        eng.load_prefix(b, kvs[b], dkvs[b], pend[b])
    dev = torch.device("cuda")
    slots = torch.arange(B, dtype=torch.int32, device=dev)
    toks = [[] for _ in range(B)]      # committed tokens t_0, t_1, ...
    bgpu = [[] for _ in range(B)]      # b row of the verify row that produced each of them
    steps, accepted = 0, 0
    first = True
    while min(len(t) for t in toks) < N_TOK:
        if first:
            cand = torch.tensor([[p] for p in pend], dtype=torch.int32, device=dev)
        else:
            cand = torch.empty(B, K + 1, dtype=torch.int32, device=dev)
            eng.draft_step(slots, K, cand)
        Kc = cand.shape[1] - 1
        vt = torch.empty(B, Kc + 1, dtype=torch.int32, device=dev)
        acc = torch.empty(B, dtype=torch.int32, device=dev)
        eng.verify_step(slots, cand, vt, acc)
        brows = eng.read_workspace(F.WS_B, (B * (Kc + 1), shape.hidden), torch.bfloat16)
        com = torch.empty(B, Kc + 1, dtype=torch.int32, device=dev)
        nc = torch.empty(B, dtype=torch.int32, device=dev)
        eng.accept_commit(slots, com, nc)
        eng.sync()
        for b in range(B):
            m = int(acc[b]) if Kc > 0 else 0
            assert int(nc[b]) == m + 1
            for j in range(m + 1):
                # committed token j of this step is v_j, produced by verify row j
                assert int(com[b, j]) == int(vt[b, j])
                toks[b].append(int(vt[b, j]))
                bgpu[b].append(brows[b * (Kc + 1) + j])
            if not first:
                accepted += m
        steps += 0 if first else 1
        first = False
    eng.close()
    assert accepted > 0, "the tuned draft head should get drafts accepted"

    # ---- oracle: plain greedy decoding from the same prefix, one token per step
    model = O.Verifier(vw)
    caches = [O.SeqCache.from_prefix(kvs[b], pend[b]) for b in range(B)]
    compared = 0
    alive = [True] * B
    for i in range(N_TOK):
        cand = [[c.pending] for c in caches]
        vo = O.verify(model, caches, cand, rb=True)
        for b in range(B):
            if not alive[b]:
                continue
            b_ref = vo.b[b, 0]
            assert rel_err(bgpu[b][i], b_ref) < REL_TOL, (b, i)
            margin = argmax_margin(vw.lm_head, bgpu[b][i][None], b_ref[None])[0]
            if float(vo.v_gap[b, 0]) <= margin:
                alive[b] = False
                continue
            assert toks[b][i] == int(vo.v[b, 0]), (b, i)
            compared += 1
        O.commit(caches, vo, cand)
    print(f"[parity] 12-layer speculative stream vs oracle greedy: {compared} tokens compared over {B} "
          f"sequences, {steps} speculative steps, {accepted} drafts accepted")
    assert compared >= 16
