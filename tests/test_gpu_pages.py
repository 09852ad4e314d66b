"""Paged KV cache: the step does not depend on where a sequence's pages sit in the pool.  The
same speculative loop (the FastMTP head's drafts, verify, commit) runs once with every
sequence's pages contiguous and once with all pages of the pool handed out in a seeded random
order, so that the sequences' pages interleave; committed tokens and accept lengths must be
identical, and so must the committed K/V rows read back through each run's block table
(bit for bit: only the page addresses differ between the runs)."""
import numpy as np
import pytest
import torch

import synth_inputs as S
from paper_2609_03181_gb300 import fastmtp as F

pytestmark = pytest.mark.gpu

SHAPE = S.ModelShape(n_layers=2, vocab=4096)
B, K, N_TOK = 4, 3, 12


def load_prefix_paged(eng, slot, kv, dkv, pending, bt):
    """The verifier and draft prefixes of one sequence into the pages bt[0], bt[1], ..."""
    ps = eng.page_size
    ctx = kv.shape[2]
    n = (ctx + ps - 1) // ps
    pad = n * ps - ctx
    src = torch.nn.functional.pad(kv.to(eng.device), (0, 0, 0, 0, 0, pad))
    src = src.reshape(kv.shape[0], 2, n, ps, kv.shape[3], kv.shape[4]).permute(0, 2, 1, 4, 3, 5)
    dsrc = torch.nn.functional.pad(dkv.to(eng.device), (0, 0, 0, 0, 0, pad))
    dsrc = dsrc.reshape(2, n, ps, dkv.shape[2], dkv.shape[3]).permute(1, 0, 3, 2, 4)
    for i in range(n):
        eng.kv_pool[:, bt[i]] = src[:, i]
        eng.dkv_pool[bt[i]] = dsrc[i]
    torch.cuda.synchronize(eng.device)
    eng.reset_seq(slot, ctx, bt, pending)


def run(eng, tables, kvs, dkvs, pend):
    dev = torch.device("cuda")
    for b in range(B):
        load_prefix_paged(eng, b, kvs[b], dkvs[b], pend[b], tables[b])
    slots = torch.arange(B, dtype=torch.int32, device=dev)
    out, ms, first = [[] for _ in range(B)], [], True
    while min(len(o) for o in out) < N_TOK:
        if first:
            cand = torch.tensor([[eng.seq_state(b)[1]] for b in range(B)], dtype=torch.int32, device=dev)
        else:
            cand = torch.empty(B, K + 1, dtype=torch.int32, device=dev)
            eng.draft_step(slots, K, cand)
        kc = cand.shape[1] - 1
        vt = torch.empty(B, kc + 1, dtype=torch.int32, device=dev)
        acc = torch.empty(B, dtype=torch.int32, device=dev)
        eng.verify_step(slots, cand, vt, acc)
        com = torch.empty(B, kc + 1, dtype=torch.int32, device=dev)
        nc = torch.empty(B, dtype=torch.int32, device=dev)
        eng.accept_commit(slots, com, nc)
        eng.sync()
        for b in range(B):
            out[b].extend(com[b, : int(nc[b])].tolist())
        ms.extend(acc.tolist() if kc > 0 else [])
        first = False
    # every committed verifier K/V row, read back through this run's block table
    ps = eng.page_size
    rows = []
    for b in range(B):
        n_ctx = eng.seq_state(b)[0]
        pos = torch.arange(n_ctx)
        pages = torch.tensor(tables[b])[pos // ps]
        rows.append(eng.kv_pool[:, pages.to(eng.device), :, :, (pos % ps).to(eng.device), :].cpu())
    return out, ms, rows


def test_step_does_not_depend_on_page_placement():
    seed = 29
    vw, dw, _ = S.successor_weights(SHAPE, seed, 7.0)
    ctx = [int(c) for c in S.integers(seed, "ctx", B, 100, 300)]
    kvs = [S.kv_prefix(seed, b, SHAPE.n_layers, ctx[b], SHAPE.n_heads, SHAPE.head_dim) for b in range(B)]
    dkvs = [S.draft_kv_prefix(seed, b, ctx[b], SHAPE.n_heads, SHAPE.head_dim) for b in range(B)]
    pend = [int(x) for x in S.integers(seed, "pending", B, 0, SHAPE.vocab - 1)]
    eng = F.Engine(vw, dw, max_batch=B, K_max=K, max_ctx=max(ctx) + 2 * N_TOK + 16, page_size=64)
    try:
        contiguous = [eng.block_table(b) for b in range(B)]
        perm = np.random.default_rng(seed).permutation(eng.n_pages).tolist()
        scattered = [perm[b * eng.max_pages:(b + 1) * eng.max_pages] for b in range(B)]
        assert any(t != sorted(t) or t[0] != b * eng.max_pages for b, t in enumerate(scattered))
        out_a, ms_a, rows_a = run(eng, contiguous, kvs, dkvs, pend)
        out_b, ms_b, rows_b = run(eng, scattered, kvs, dkvs, pend)
        assert out_a == out_b
        assert ms_a == ms_b
        assert max(ms_a) > 0                                   # drafts were accepted: the K/V rows moved
        for b in range(B):
            assert torch.equal(rows_a[b], rows_b[b]), b
    finally:
        eng.close()
