"""verify_step + accept_commit through the C ABI against the fp64 oracle (storage-rounding
mode): one decoder layer at the paper's widths (B=1, K=3, context 512, full vocabulary), then
the 12-layer decoder (B=8, K=3, contexts U[768,1024] with a 256-token synthetic visual prefix).

Rules: b = N_o(h_L) and the committed K/V within max relative error 2e-2; router experts,
verifier tokens and accept lengths bit-exact where the oracle's fp64 top-2 margin exceeds 1e-3."""
import numpy as np
import pytest
import torch

import oracle as O
import synth_inputs as S
from paper_2609_03181_gb300 import fastmtp as F
from tests.gpu_util import REL_TOL, GAP, rel_err, seq_prefixes, make_drafts, index_parity, argmax_margin

pytestmark = pytest.mark.gpu


def run_verify_case(shape, seed, ctx_lens, K, gain_std=0.1, check=None, zipf_s=None, rb=True, min_keep=None,
                    fp8=False, rel_tol=REL_TOL):
    """One verify_step + accept_commit of len(ctx_lens) sequences on the GPU; the sequences in
    `check` (default: all) are compared with the oracle (storage-rounding mode if `rb`, else the
    plain fp64 definition), the others get uniform random drafts and only fill the batch.
    `fp8` runs the fp8-expert variant on both sides; `rel_tol` replaces the 2e-2 rule for it.
    `min_keep` is the least number of checked rows that must stay comparable through every layer
    (default: all of them when fewer than four sequences are checked, else all but two
    sequences' rows).  Prints the comparison counts and returns them."""
    B = len(ctx_lens)
    check = list(range(B)) if check is None else list(check)
    vw = S.verifier_weights(shape, seed, gain_std=gain_std, zipf_s=zipf_s)
    if fp8:   # the fp8-expert variant: e4m3 expert matrices with per-row scales, on both sides
        vw = S.quantize_experts_fp8(vw)
    dw = S.draft_weights(shape, seed, gain_std=gain_std)
    model = O.Verifier(vw)
    kvs, dkvs = seq_prefixes(shape, seed, ctx_lens)
    pend = S.integers(seed, "pending", B, 0, shape.vocab - 1)
    caches = [O.SeqCache.from_prefix(kvs[b], int(pend[b])) for b in check]
    cand_chk = make_drafts(model, caches, K, seed)
    other = S.integers(seed, "draft.other", B * K, 0, shape.vocab - 1).reshape(B, K)
    cand = [[int(pend[b])] + [int(t) for t in other[b]] for b in range(B)]
    for j, b in enumerate(check):
        cand[b] = cand_chk[j]
    ref = O.verify(model, caches, cand_chk, rb=rb, keep_hidden=True)

    eng = F.Engine(vw, dw, max_batch=B, K_max=max(K, 3), max_ctx=max(ctx_lens) + 8, page_size=64, expert_fp8=fp8)
    for b in range(B):
        eng.load_prefix(b, kvs[b], dkvs[b], int(pend[b]))
    dev = torch.device("cuda")
    slots = torch.arange(B, dtype=torch.int32, device=dev)
    cand_d = torch.tensor(cand, dtype=torch.int32, device=dev)
    vt = torch.empty(B, K + 1, dtype=torch.int32, device=dev)
    acc = torch.empty(B, dtype=torch.int32, device=dev)
    eng.verify_step(slots, cand_d, vt, acc)
    eng.sync()
    R = K + 1
    rows = [b * R + r for b in check for r in range(R)]   # GPU rows of the checked sequences
    T = len(rows)
    b_all = eng.read_workspace(F.WS_B, (B * R, shape.hidden), torch.bfloat16)
    b_gpu = b_all[rows]
    ridx = eng.read_workspace(F.WS_ROUTE_IDX, (shape.n_layers, eng.max_batch * (eng.K_max + 1), shape.top_k),
                              torch.int32)
    # Routing: bit-exact wherever the oracle's 6th/7th probability margin exceeds 1e-3.  A row
    # whose expert set differs below the margin (a legitimate near-tie) leaves the comparison of
    # hidden states from then on, together with the later candidates of its sequence (they
    # attend to its K/V); such rows are counted.
    # Per layer, the router probabilities of the selected experts of every row still comparable
    # (its selections and those of the earlier rows of its sequence equal so far) are a check of
    # the layer's hidden state: within 2e-2 of the oracle's, relative to the row's largest.
    gate_gpu = eng.read_workspace(F.WS_ROUTE_GATE, (shape.n_layers, eng.max_batch * (eng.K_max + 1), shape.top_k),
                                  torch.float32)
    diverged = np.zeros(T, dtype=bool)
    near_ties = 0
    div_per_layer = []
    for l in range(shape.n_layers):
        gi = ridx[l, rows].numpy()
        g = np.sort(gi, -1)
        r = np.sort(ref.route_idx[l].numpy(), -1)
        live = ~diverged
        n_ok, n_skip, n_bad = index_parity(g[live], r[live], ref.route_gap[l].numpy()[live])
        near_ties += n_skip
        assert n_bad == 0, f"layer {l}: {n_bad} router mismatches over {n_ok} rows"
        same = live & ~(g != r).any(-1)
        for i in np.nonzero(same)[0]:
            og = np.argsort(gi[i])
            orf = np.argsort(ref.route_idx[l][i].numpy())
            e = rel_err(gate_gpu[l, rows[i]][og], ref.route_gate[l][i][orf])
            assert e < rel_tol, f"layer {l} row {i}: router probability rel err {e:.3g}"
        differ = (g != r).any(-1) & ~diverged
        div_per_layer.append(int(differ.sum()))
        for row in np.nonzero(differ)[0]:
            seq = row // R
            diverged[row:(seq + 1) * R] = True
    keep = ~diverged
    errs = [rel_err(b_gpu[i], ref.b.reshape(T, -1)[i]) for i in range(T)]
    # bf16 storage decorrelates GPU and oracle rounding decisions over many layers (about 1%
    # hidden-state noise at 12 layers), so a router near-tie can resolve differently; such a row
    # and the later rows of its sequence leave the comparison (counted and printed)
    # default floor: every row when one to three sequences are checked, else all but the rows of
    # two sequences
    need = (T if len(check) < 4 else T - 2 * R) if min_keep is None else min_keep
    print(f"[parity] layers {shape.n_layers}, rows {T}, comparable through every layer {int(keep.sum())}, "
          f"router near-ties skipped {near_ties}, rows leaving per layer {div_per_layer}")
    assert keep.sum() >= need, f"only {keep.sum()} of {T} rows comparable (need {need})"
    assert max(e for e, k in zip(errs, keep) if k) < rel_tol, (
        f"b rel err per row {['%.3g' % e for e in errs]}, diverged rows {np.nonzero(diverged)[0].tolist()}")
    # the fp32 residual stream after the last layer, row by row
    h_gpu = eng.read_workspace(F.WS_HIDDEN, (B * R, shape.hidden), torch.float32)[rows]
    h_ref = ref.hidden[-1]
    for i in np.nonzero(keep)[0]:
        e = rel_err(h_gpu[i], h_ref[i])
        assert e < rel_tol, f"row {i}: residual stream rel err {e:.3g}"

    # verifier tokens: exact where the oracle's logit margin exceeds the noise the measured state
    # difference implies (at least 1e-3); accept lengths where all of a sequence's tokens are
    margin = argmax_margin(vw.lm_head, b_gpu, ref.b.reshape(T, -1))
    gaps = ref.v_gap.numpy().reshape(-1)
    sure = keep & (gaps > margin)
    g_tok, r_tok = vt.cpu().numpy()[check].reshape(-1), ref.v.numpy().reshape(-1)
    assert (g_tok[sure] == r_tok[sure]).all(), (
        f"token mismatch at rows {np.nonzero(sure & (g_tok != r_tok))[0].tolist()}")
    for j, bb in enumerate(check):
        rr = slice(j * R, j * R + K)
        if sure[rr].all():
            assert int(acc[bb]) == ref.m[j]

    committed = torch.empty(B, K + 1, dtype=torch.int32, device=dev)
    ncom = torch.empty(B, dtype=torch.int32, device=dev)
    eng.accept_commit(slots, committed, ncom)
    eng.sync()
    ps = eng.page_size
    for b in range(B):
        m = int(acc[b])
        assert int(ncom[b]) == m + 1
        toks = committed[b].tolist()
        assert toks[:m + 1] == cand[b][1:m + 1] + [int(vt[b, m])] and all(t == -1 for t in toks[m + 1:])
        ln, pending = eng.seq_state(b)
        assert ln == ctx_lens[b] + m + 1 and pending == int(vt[b, m])
    for j, b in enumerate(check):
        m = int(acc[b])
        bt = eng.block_table(b)
        if m != ref.m[j]:
            continue
        for l in range(shape.n_layers):
            for r in range(m + 1):
                if diverged[j * R + r]:
                    continue
                p = ctx_lens[b] + r
                page, off = bt[p // ps], p % ps
                k_gpu = eng.kv_pool[l, page, 0, :, off, :].cpu()
                v_gpu = eng.kv_pool[l, page, 1, :, off, :].cpu()
                assert rel_err(k_gpu, ref.new_k[j][l][r]) < rel_tol
                assert rel_err(v_gpu, ref.new_v[j][l][r]) < rel_tol
    eng.close()
    print(f"[parity] verifier tokens compared {int(sure.sum())}, below the margin {int((~sure).sum())}")
    return {"rows": T, "kept": int(keep.sum()), "near_ties": near_ties, "tokens": int(sure.sum()),
            "tokens_skipped": int((~sure).sum())}


def test_verify_one_layer_b1_ctx512():
    shape = S.ModelShape(n_layers=1)
    run_verify_case(shape, 0, [512], K=3)


def test_verify_one_layer_against_plain_definition():
    """The same one-layer step against the oracle without storage rounding (rb=False: fp64
    everywhere between the bf16 weights and inputs), so that a precision shortcut the rounding
    mode happened to copy would still show: b and the committed K/V within 2e-2, routing and
    tokens exact above the margins."""
    shape = S.ModelShape(n_layers=1)
    run_verify_case(shape, 0, [512], K=3, rb=False)
    run_verify_case(S.ModelShape(n_layers=2, vocab=4096), 5, [0, 63, 200, 777], K=3, rb=False)


def test_verify_ragged_small_contexts():
    """Empty committed context, contexts inside the first chunk and across page boundaries."""
    shape = S.ModelShape(n_layers=2, vocab=4096)
    run_verify_case(shape, 5, [0, 1, 63, 64, 129, 200], K=2)


def test_verify_twelve_layers_b8_ctx768_1024():
    shape = S.ModelShape()
    ctx = [int(c) for c in S.integers(1, "ctx", 8, 768, 1024)]
    run_verify_case(shape, 1, ctx, K=3, gain_std=0.0, min_keep=16)


def test_verify_max_batch_256():
    """The largest batch of the throughput sweep, B=256 (T=1024 candidate rows, 128-row dual
    expert items): 16 sequences spread over the batch are checked against the oracle."""
    shape = S.ModelShape(n_layers=1, vocab=4096)
    ctx = [int(c) for c in S.integers(9, "ctx", 256, 1, 160)]
    run_verify_case(shape, 9, ctx, K=3, check=range(3, 256, 16))


def test_verify_zipf_hot_experts():
    """Zipf-skewed routing (router bias -1.2 ln(rank)): the hottest experts take most of the 192
    candidate rows, so their gate/up and down tiles span several 64-row tiles and every down
    tile waits on the gate/up tiles of its own rows; 8 of the 48 sequences are checked."""
    shape = S.ModelShape(n_layers=2, vocab=4096)
    ctx = [int(c) for c in S.integers(11, "ctx", 48, 1, 300)]
    run_verify_case(shape, 11, ctx, K=3, check=range(0, 48, 6), zipf_s=1.2)
