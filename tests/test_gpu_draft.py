"""draft_step through the C ABI against the fp64 oracle's FastMTP head: the shared block
alone at the paper's widths (B=32, draft-cache context 2048, K=3; also B=1 and 8), with 1..4
rows queued per sequence (base states b ~ N(0,1), as a commit of m = 0..3 accepted drafts leaves
them).

Rules: the committed draft K/V rows and the draft states u^(k) within max relative error
2e-2; drafted tokens bit-exact at every depth whose oracle top-2 margin exceeds 1e-3 (a depth
below the margin ends the comparison of that sequence, since later depths consume its token)."""
import numpy as np
import pytest
import torch

import oracle as O
import synth_inputs as S
from paper_2609_03181_gb300 import fastmtp as F
from tests.gpu_util import REL_TOL, GAP, rel_err

pytestmark = pytest.mark.gpu


def run_draft_case(B, ctx, K, seed, vocab=129280):
    shape = S.ModelShape(n_layers=1, vocab=vocab)
    vw = S.verifier_weights(shape, seed, gain_std=0.1)
    dw = S.draft_weights(shape, seed, gain_std=0.1)
    model = O.Verifier(vw)
    dr = O.Drafter(dw, model)
    n_rows = [int(x) + 1 for x in S.integers(seed, "mrows", B, 0, K)]
    pend = [int(x) for x in S.integers(seed, "pending", B, 0, vocab - 1)]
    eng = F.Engine(vw, dw, max_batch=B, K_max=K, max_ctx=ctx + K + 8, page_size=64)
    dcs = []
    for b in range(B):
        dkv = S.draft_kv_prefix(seed, b, ctx, shape.n_heads, shape.head_dim)
        rows_b = S.normal(seed, f"brows.{b}", (n_rows[b], shape.hidden), 1.0)
        toks = [int(t) for t in S.integers(seed, f"btok.{b}", n_rows[b], 0, vocab - 1)]
        toks[-1] = pend[b]
        dc = O.DraftCache.from_prefix(dkv)
        dc.rows_b, dc.rows_tok = rows_b.double(), toks
        dcs.append(dc)
        eng.load_prefix(b, None, dkv, pend[b], ctx_len=ctx + n_rows[b])
        eng.set_draft_rows(b, rows_b, toks)
    ref = O.draft(dr, dcs, K, rb=True)
    dev = torch.device("cuda")
    slots = torch.arange(B, dtype=torch.int32, device=dev)
    cand = torch.full((B, K + 1), -5, dtype=torch.int32, device=dev)
    eng.draft_step(slots, K, cand)
    eng.sync()
    cand = cand.cpu()
    u = eng.read_workspace(F.WS_DRAFT_U, (K, B, shape.hidden), torch.bfloat16)
    checked = skipped = 0
    for b in range(B):
        assert int(cand[b, 0]) == pend[b]
        for k in range(K):
            assert rel_err(u[k, b], ref.u[b][k]) < REL_TOL, (b, k)
            if ref.gaps[b][k] <= GAP:
                skipped += 1
                break
            assert int(cand[b, k + 1]) == ref.tokens[b][k], (b, k)
            checked += 1
        # committed draft rows written at positions ctx .. ctx+n-1 (base states)
        bt = eng.block_table(b)
        for i in range(n_rows[b]):
            p = ctx + i
            page, off = bt[p // eng.page_size], p % eng.page_size
            assert rel_err(eng.dkv_pool[page, 0, :, off, :].cpu(), ref.row_k[b][i]) < REL_TOL
            assert rel_err(eng.dkv_pool[page, 1, :, off, :].cpu(), ref.row_v[b][i]) < REL_TOL
    eng.close()
    assert checked > 0
    return checked, skipped


def test_draft_block_b32_ctx2048():
    run_draft_case(B=32, ctx=2048, K=3, seed=2)


@pytest.mark.parametrize("B", [1, 8])
def test_draft_small_batch(B):
    """The small batches of the latency-bound regime (one 16-row activation box, cluster
    split-K GEMMs), same rules."""
    run_draft_case(B=B, ctx=2048, K=3, seed=4 + B)


def test_draft_small_context_deep_chain():
    """Short context (the chain's tentative rows are most of the keys) and K = 5."""
    run_draft_case(B=3, ctx=5, K=5, seed=12, vocab=2048)
