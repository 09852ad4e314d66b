"""Pins of the fp64 oracle against what the paper and the mathematics fix (CPU only).

Each test checks an oracle function against something other than its own formula: a library
routine computing the same textbook operation, a closed form, brute force over a tiny input,
an invariant the method guarantees (causality, incremental == parallel, losslessness of greedy
verification), or numbers printed in the paper (tests/golden/)."""
import itertools
import json
import math
import os

import numpy as np
import pytest
import torch
import torch.nn.functional as F

import oracle as O
import synth_inputs as S

GOLD = os.path.join(os.path.dirname(__file__), "golden")
F64 = torch.float64

TINY = S.ModelShape(hidden=12, n_heads=2, head_dim=4, n_layers=2, n_experts=5, top_k=2, n_shared=1,
                    expert_inter=6, draft_inter=10, vocab=40, rope_theta=10000.0, max_position=512)


def tiny_model(seed=0, std=0.3, shape=TINY, gain_std=0.2):
    w = S.verifier_weights(shape, seed, std=std, gain_std=gain_std)
    return O.Verifier(w)


def tiny_caches(shape, seed, B, ctx_lo, ctx_hi, pending=None):
    ctxs = S.integers(seed, "ctx", B, ctx_lo, ctx_hi)
    toks = S.integers(seed, "pend", B, 0, shape.vocab - 1) if pending is None else pending
    return [O.SeqCache.from_prefix(S.kv_prefix(seed, b, shape.n_layers, int(ctxs[b]), shape.n_heads,
                                               shape.head_dim), int(toks[b])) for b in range(B)]


# ----------------------------------------------------------------------------- precision

def test_round_bf16_matches_torch_rne_on_fp32_inputs():
    x = torch.randn(200000, generator=torch.Generator().manual_seed(1), dtype=torch.float32) * 3
    ref = x.to(torch.bfloat16).to(F64)          # torch's fp32 -> bf16 is round-to-nearest-even
    got = O.round_bf16(x.to(F64))
    assert torch.equal(got, ref)


def test_round_bf16_ties_and_single_step():
    # 1 + 2^-8 is halfway between 1 and 1 + 2^-7: ties to even -> 1
    assert O.round_bf16(torch.tensor([1 + 2 ** -8], dtype=F64)).item() == 1.0
    # 1 + 3*2^-8 is halfway between 1+2^-7 and 1+2^-6: even mantissa is 1+2^-6
    assert O.round_bf16(torch.tensor([1 + 3 * 2 ** -8], dtype=F64)).item() == 1 + 2 ** -6
    # just above a tie rounds up (would be lost by rounding through fp32 first)
    v = 1 + 2 ** -8 + 2 ** -40
    assert O.round_bf16(torch.tensor([v], dtype=F64)).item() == 1 + 2 ** -7
    assert O.round_bf16(torch.tensor([0.0, -0.0], dtype=F64)).abs().sum().item() == 0.0


# ----------------------------------------------------------------------------- RMSNorm

def test_rms_norm_closed_forms():
    # [3, 4]: mean square 12.5
    y = O.rms_norm(torch.tensor([3.0, 4.0], dtype=F64), torch.tensor([1.0, 2.0]), 0.0)
    assert torch.allclose(y, torch.tensor([3 / math.sqrt(12.5), 8 / math.sqrt(12.5)], dtype=F64))
    # constant vector c with eps: c / sqrt(c^2 + eps) * gain
    c, eps = 0.01, 1e-3
    y = O.rms_norm(torch.full((7,), c, dtype=F64), torch.full((7,), 1.5), eps)
    assert torch.allclose(y, torch.full((7,), 1.5 * c / math.sqrt(c * c + eps), dtype=F64))


def test_rms_norm_matches_library():
    g = torch.Generator().manual_seed(3)
    x = torch.randn(5, 33, generator=g, dtype=F64)
    w = torch.randn(33, generator=g, dtype=F64)
    ref = F.rms_norm(x, (33,), w, eps=1e-6)
    assert torch.allclose(O.rms_norm(x, w, 1e-6), ref, rtol=1e-12, atol=1e-12)


# ----------------------------------------------------------------------------- RoPE

def _rope_complex(x, pos, theta):
    """Independent formulation: pair (i, i+hd/2) as a complex number times e^{i*pos*w_i}."""
    hd = x.shape[-1]
    half = hd // 2
    w = torch.tensor([1.0 / theta ** (2 * i / hd) for i in range(half)], dtype=F64)
    z = torch.complex(x[..., :half], x[..., half:])
    rot = torch.polar(torch.ones(len(pos), half, dtype=F64), torch.as_tensor(pos, dtype=F64)[:, None] * w)
    r = z * rot[:, None, :]
    return torch.cat([r.real, r.imag], -1)


def test_rope_equals_complex_rotation():
    g = torch.Generator().manual_seed(4)
    x = torch.randn(6, 3, 8, generator=g, dtype=F64)
    pos = [0, 1, 5, 100, 4095, 32767]
    assert torch.allclose(O.rope(x, torch.tensor(pos), 1e6), _rope_complex(x, pos, 1e6), atol=1e-12)


def test_rope_hand_value_and_relative_position():
    # hd=2: a plain 2-D rotation by pos radians
    y = O.rope(torch.tensor([[[1.0, 0.0]]], dtype=F64), torch.tensor([1]), 1e6)
    assert torch.allclose(y, torch.tensor([[[math.cos(1), math.sin(1)]]], dtype=F64))
    # <rope(q, m), rope(k, n)> depends only on m - n; position 0 is the identity
    g = torch.Generator().manual_seed(5)
    q, k = torch.randn(1, 1, 16, generator=g, dtype=F64), torch.randn(1, 1, 16, generator=g, dtype=F64)
    d = lambda m, n: (O.rope(q, torch.tensor([m]), 1e4) * O.rope(k, torch.tensor([n]), 1e4)).sum()
    assert abs(d(7, 3) - d(104, 100)) < 1e-10
    assert torch.equal(O.rope(q, torch.tensor([0]), 1e4), q)


# ----------------------------------------------------------------------------- attention

def test_attention_matches_library_sdpa():
    g = torch.Generator().manual_seed(6)
    n, R, H, hd = 23, 4, 3, 8
    k = torch.randn(n, H, hd, generator=g, dtype=F64)
    v = torch.randn(n, H, hd, generator=g, dtype=F64)
    q = torch.randn(R, H, hd, generator=g, dtype=F64)
    qpos = [19, 20, 21, 22]
    mask = torch.tensor([[j <= p for j in range(n)] for p in qpos])
    ref = F.scaled_dot_product_attention(q.transpose(0, 1), k.transpose(0, 1), v.transpose(0, 1),
                                         attn_mask=mask[None]).transpose(0, 1)
    assert torch.allclose(O.attention(q, qpos, k, v), ref, atol=1e-12)


def test_attention_special_cases():
    g = torch.Generator().manual_seed(7)
    v = torch.randn(5, 2, 4, generator=g, dtype=F64)
    q = torch.randn(1, 2, 4, generator=g, dtype=F64)
    # a single visible key (empty committed context): output is that key's value
    out = O.attention(q, [0], torch.randn(5, 2, 4, generator=g, dtype=F64), v)
    assert torch.allclose(out[0], v[0])
    # identical keys: uniform weights, output is the mean of the visible values
    k = torch.randn(1, 2, 4, generator=g, dtype=F64).expand(5, 2, 4)
    out = O.attention(q, [3], k, v)
    assert torch.allclose(out[0], v[:4].mean(0))


# ----------------------------------------------------------------------------- FFN / router

def test_silu_and_swiglu_match_library():
    g = torch.Generator().manual_seed(8)
    x = torch.randn(9, generator=g, dtype=F64)
    assert torch.allclose(O.silu(x), F.silu(x))
    xs = torch.randn(3, 12, generator=g, dtype=F64)
    wgu = torch.randn(14, 12, generator=g, dtype=F64)
    wd = torch.randn(12, 7, generator=g, dtype=F64)
    ref = F.linear(F.silu(F.linear(xs, wgu[:7])) * F.linear(xs, wgu[7:]), wd)
    assert torch.allclose(O.swiglu(xs, wgu, wd, rb=False), ref)


def test_router_topk_brute_force():
    g = torch.Generator().manual_seed(9)
    E, k = 6, 3
    x = torch.randn(20, 4, generator=g, dtype=F64)
    wr = torch.randn(E, 4, generator=g, dtype=F64)
    idx, gates, p, gap = O.router_topk(x, wr, k)
    logits = x @ wr.T
    for t in range(20):
        pt = [math.exp(l) for l in logits[t].tolist()]
        pt = [a / sum(pt) for a in pt]
        best = max(itertools.combinations(range(E), k), key=lambda c: sum(pt[i] for i in c))
        assert sorted(idx[t].tolist()) == sorted(best)
        assert idx[t].tolist() == sorted(best, key=lambda i: -pt[i])
        assert torch.allclose(gates[t], torch.tensor([pt[i] for i in idx[t].tolist()], dtype=F64))
        srt = sorted(pt, reverse=True)
        assert abs(gap[t].item() - (srt[k - 1] - srt[k])) < 1e-12


def test_router_ties_go_to_lower_expert_and_bias_shifts_logits():
    x = torch.ones(1, 2, dtype=F64)
    wr = torch.tensor([[0.0, 0.0], [1.0, 0.0], [0.0, 0.0], [1.0, 0.0], [0.0, 0.0]], dtype=F64)
    idx, _, _, gap = O.router_topk(x, wr, 3)
    assert idx[0].tolist() == [1, 3, 0] and gap[0].item() == 0.0
    idx, _, _, _ = O.router_topk(x, wr, 2, bias=torch.tensor([5.0, 0, 0, 0, 0]))
    assert idx[0].tolist() == [0, 1]


def _moe_once(model, x, rb=False):
    lw = model.w.layers[0]
    return O.model._moe(model, lw, x, rb)


def test_moe_topk_equals_E_is_dense_probability_weighted_sum():
    sh = TINY.replace(n_experts=3, top_k=3, n_shared=1)
    model = tiny_model(1, shape=sh)
    lw = model.w.layers[0]
    x = torch.randn(4, sh.hidden, generator=torch.Generator().manual_seed(2), dtype=F64)
    y, idx, gates, _ = _moe_once(model, x)
    p = torch.softmax(x @ lw.router.to(F64).T, -1)
    dense = sum(p[:, e:e + 1] * O.swiglu(x, lw.w_gate_up[e], lw.w_down[e], False) for e in range(3))
    dense = dense + O.swiglu(x, lw.shared_gate_up[0], lw.shared_down[0], False)
    assert torch.allclose(y, dense, atol=1e-12)


def test_moe_single_expert_top1_is_plain_swiglu_plus_shared():
    sh = TINY.replace(n_experts=1, top_k=1, n_shared=2)
    model = tiny_model(2, shape=sh)
    lw = model.w.layers[0]
    x = torch.randn(3, sh.hidden, generator=torch.Generator().manual_seed(3), dtype=F64)
    y, idx, gates, _ = _moe_once(model, x)
    assert torch.all(gates == 1.0)
    ref = F.linear(F.silu(F.linear(x, lw.w_gate_up[0, :6].to(F64))) * F.linear(x, lw.w_gate_up[0, 6:].to(F64)),
                   lw.w_down[0].to(F64))
    for j in range(2):
        ref = ref + F.linear(F.silu(F.linear(x, lw.shared_gate_up[j, :6].to(F64))) *
                             F.linear(x, lw.shared_gate_up[j, 6:].to(F64)), lw.shared_down[j].to(F64))
    assert torch.allclose(y, ref, atol=1e-12)


def test_moe_is_invariant_to_expert_relabelling():
    model = tiny_model(3)
    lw = model.w.layers[0]
    x = torch.randn(6, TINY.hidden, generator=torch.Generator().manual_seed(4), dtype=F64)
    y0 = _moe_once(model, x)[0]
    perm = torch.tensor([3, 0, 4, 1, 2])
    lw.router, lw.w_gate_up, lw.w_down = lw.router[perm], lw.w_gate_up[perm], lw.w_down[perm]
    assert torch.allclose(_moe_once(model, x)[0], y0, atol=1e-12)


# ----------------------------------------------------------------------------- greedy argmax

def test_argmax_with_gap_hand_values():
    """v_r = argmax of each row, the lowest id among equal maxima (the reading for ties), and the
    margin top-1 minus top-2 taken on the row's own values (0 for a tie).  Expected numbers are
    written out by hand, not produced by another argmax."""
    logits = torch.tensor([
        [1.0, 3.0, 3.0, 2.0],            # tie of ids 1 and 2 at the maximum -> 1, margin 0
        [5.0, 1.0, 4.5, -2.0],           # clear maximum at id 0, runner-up 4.5 -> margin 0.5
        [-1.0, -1.0, -1.0, -1.0],        # all equal -> id 0, margin 0
        [0.25, 0.75, 0.5, 0.75 - 2.0 ** -20],   # near tie resolved by value -> id 1, margin 2^-20
        [-7.0, -3.0, -3.5, -9.0],        # negative values -> id 1, margin 0.5
        [2.0, 0.0, 0.0, 2.0],            # tie of the first and the last id -> 0, margin 0
    ], dtype=F64)
    v, gap = O.argmax_with_gap(logits)
    assert v.tolist() == [1, 0, 0, 1, 1, 0]
    assert gap.tolist() == [0.0, 0.5, 0.0, 2.0 ** -20, 0.5, 0.0]


def test_verify_argmax_tie_goes_to_lower_token():
    """Through verify(): with every layer the identity (zero W_o and down projections) the state
    is b = N_o(E[x]); making W_lm rows 29 and 7 equal to a scaled copy of b puts both ids at
    the exact maximum, and the verifier must answer 7 with margin 0; with row 29 scaled up by
    2^-7 it must answer 29."""
    model = tiny_model(12)
    for lw in model.w.layers:
        lw.wo = torch.zeros_like(lw.wo)
        lw.w_down = torch.zeros_like(lw.w_down)
        lw.shared_down = torch.zeros_like(lw.shared_down)
    caches = tiny_caches(TINY, 12, 1, 3, 3)
    x = caches[0].pending
    b = F.rms_norm(model.w.embed[x].to(F64), (TINY.hidden,), model.w.final_norm.to(F64), eps=TINY.rms_eps)
    row = (b * 4).to(torch.bfloat16)     # logit ~4 |b|^2 >> every random row's logit
    lm = model.w.lm_head.clone()
    lm[7] = row
    lm[29] = row
    model.w.lm_head = lm
    model._lm = None
    out = O.verify(model, caches, [[x]], rb=False)
    assert int(out.v[0, 0]) == 7 and float(out.v_gap[0, 0]) == 0.0
    lm[29] = (row.to(F64) * (1 + 2 ** -7)).to(torch.bfloat16)
    model._lm = None
    out = O.verify(model, caches, [[x]], rb=False)
    assert int(out.v[0, 0]) == 29 and float(out.v_gap[0, 0]) > 0.0


# ----------------------------------------------------------------------------- acceptance

@pytest.mark.parametrize("K", [1, 2, 3, 4])
def test_accept_length_all_match_patterns(K):
    """Eq. of Sec. 3.1 over all 2^K match masks: m = index of the first mismatch (K if none),
    committed = x^_{1:m} then v_{m+1}, so 1 <= committed <= K+1."""
    for mask in itertools.product([True, False], repeat=K):
        v = list(range(100, 100 + K + 1))
        drafts = [v[s] if mask[s] else v[s] + 1000 for s in range(K)]
        m = O.accept_length(drafts, v)
        first_bad = next((s for s in range(K) if not mask[s]), K)
        assert m == first_bad and 0 <= m <= K
        committed = drafts[:m] + [v[m]]
        assert 1 <= len(committed) <= K + 1 and committed[-1] == v[m]


# ----------------------------------------------------------------------------- decoder invariants

def test_layer_with_zero_output_projections_is_identity():
    """With W_o and every down projection zero, every layer is the identity on the residual
    stream, so b = N_o(E[x]) and v = argmax W_lm N_o(E[x]) (checked without the oracle's code)."""
    model = tiny_model(4)
    for lw in model.w.layers:
        lw.wo = torch.zeros_like(lw.wo)
        lw.w_down = torch.zeros_like(lw.w_down)
        lw.shared_down = torch.zeros_like(lw.shared_down)
    caches = tiny_caches(TINY, 4, 2, 3, 9)
    cand = [[c.pending, 7, 8] for c in caches]
    out = O.verify(model, caches, cand, rb=False)
    e = model.w.embed[torch.tensor(cand).flatten()].to(F64)
    b = F.rms_norm(e, (TINY.hidden,), model.w.final_norm.to(F64), eps=TINY.rms_eps)
    assert torch.allclose(out.b.reshape(-1, TINY.hidden), b, atol=1e-12)
    assert torch.equal(out.v.flatten(), (b @ model.w.lm_head.to(F64).T).argmax(-1))


def test_verify_is_causal_and_incremental_equals_parallel():
    """Row r of a verify pass depends only on candidates 0..r; verifying K+1 candidates in one
    pass equals feeding them one at a time through the committed cache (the property that
    makes greedy verification lossless)."""
    model = tiny_model(5)
    caches = tiny_caches(TINY, 5, 2, 4, 11)
    cand = [[c.pending, 3, 17, 22] for c in caches]
    full = O.verify(model, [O.SeqCache(list(c.k), list(c.v), c.pending) for c in caches], cand, rb=False)
    alt = [[c.pending, 3, 17, 5] for c in caches]
    part = O.verify(model, [O.SeqCache(list(c.k), list(c.v), c.pending) for c in caches], alt, rb=False)
    assert torch.allclose(full.b[:, :3], part.b[:, :3], atol=1e-12)
    assert not torch.allclose(full.b[:, 3], part.b[:, 3])
    # one candidate at a time
    inc = [O.SeqCache(list(c.k), list(c.v), c.pending) for c in caches]
    for r in range(4):
        step = O.verify(model, inc, [[cand[b][r]] for b in range(2)], rb=False)
        assert torch.allclose(step.b[:, 0], full.b[:, r], atol=1e-10)
        for b, c in enumerate(inc):
            for l in range(TINY.n_layers):
                c.k[l] = torch.cat([c.k[l], step.new_k[b][l]], 0)
                c.v[l] = torch.cat([c.v[l], step.new_v[b][l]], 0)
            if r < 3:
                c.pending = cand[b][r + 1]


def test_verify_is_invariant_to_head_relabelling():
    model = tiny_model(6)
    caches = tiny_caches(TINY, 6, 1, 5, 5)
    cand = [[caches[0].pending, 1, 2]]
    ref = O.verify(model, caches, cand, rb=False).b
    H, hd, d = TINY.n_heads, TINY.head_dim, TINY.hidden
    for lw in model.w.layers:
        q, k, v = lw.wqkv.reshape(3, H, hd, d).unbind(0)
        lw.wqkv = torch.stack([q.flip(0), k.flip(0), v.flip(0)]).reshape(3 * H * hd, d)
        lw.wo = lw.wo.reshape(d, H, hd).flip(1).reshape(d, H * hd)
    for c in caches:
        c.k = [t.flip(1) for t in c.k]
        c.v = [t.flip(1) for t in c.v]
    assert torch.allclose(O.verify(model, caches, cand, rb=False).b, ref, atol=1e-12)


def _clone(caches):
    return [O.SeqCache(list(c.k), list(c.v), c.pending) for c in caches]


@pytest.mark.parametrize("rb", [False, True])
def test_speculative_equals_greedy_for_any_drafts(rb):
    """Losslessness (Sec. 3.1): the committed stream equals plain greedy decoding for drafts that
    are all right, all wrong, or random."""
    model = tiny_model(7, std=0.5)
    base = tiny_caches(TINY, 7, 3, 2, 8)
    n, K = 12, 3
    greedy = O.greedy_decode(model, _clone(base), n + K + 2, rb)
    assert greedy == O.greedy_decode(model, _clone(base), n + K + 2, rb)  # deterministic

    def oracle_drafts(step, done):
        # the pending token is greedy[b][len(done[b]) - 1]; the right drafts follow it
        return [greedy[b][len(done[b]):len(done[b]) + K] for b in range(len(done))]

    rng = np.random.default_rng(0)
    sources = {
        "right": oracle_drafts,
        "wrong": lambda step, pend: [[(t + 1) % TINY.vocab for t in d] for d in oracle_drafts(step, pend)],
        "random": lambda step, pend: [list(rng.integers(0, TINY.vocab, K)) for _ in pend],
    }
    for name, fn in sources.items():
        st = O.DecodeStats()
        got = O.speculative_decode(model, _clone(base), n, K, draft_fn=fn, rb=rb, stats=st)
        assert got == [g[:n] for g in greedy], name
        if name == "right":
            assert st.accept_hist[K] == sum(st.accept_hist)
        if name == "wrong":
            assert st.accept_hist[0] == sum(st.accept_hist)


# ----------------------------------------------------------------------------- draft head

def _tiny_drafter(seed, model, gain_std=0.2):
    return O.Drafter(S.draft_weights(model.s, seed, std=0.3, gain_std=gain_std), model)


def _dcaches(shape, caches, seed):
    return [O.DraftCache.from_prefix(S.draft_kv_prefix(seed, b, c.ctx, shape.n_heads, shape.head_dim))
            for b, c in enumerate(caches)]


def test_identity_draft_block_closed_form():
    """With B_theta's W_o and W_down zero the block is the identity on z, so
    x^_1 = argmax W_lm N_o(P[N_e(E x_{j+1}); N_h(b_j)]) and deeper depths feed u back in."""
    model = tiny_model(8)
    dr = _tiny_drafter(8, model)
    dr.dw.wo = torch.zeros_like(dr.dw.wo)
    dr.dw.w_down = torch.zeros_like(dr.dw.w_down)
    caches = tiny_caches(TINY, 8, 2, 3, 6)
    dcs = _dcaches(TINY, caches, 8)
    vo = O.verify(model, caches, [[c.pending] for c in caches], rb=False)
    O.commit(caches, vo, [[c.pending] for c in caches], dcs)
    rows_b = [dc.rows_b.clone() for dc in dcs]
    rows_t = [list(dc.rows_tok) for dc in dcs]
    out = O.draft(dr, dcs, 3, rb=False)
    d = TINY.hidden
    rn = lambda x, g: F.rms_norm(x, (d,), g.to(F64), eps=TINY.rms_eps)
    E, W = model.w.embed.to(F64), model.w.lm_head.to(F64)
    for b in range(2):
        a, tok = rows_b[b][-1].to(F64), rows_t[b][-1]
        for k in range(3):
            z = F.linear(torch.cat([rn(E[tok], dr.dw.enorm), rn(a, dr.dw.hnorm)]), dr.dw.eh_proj.to(F64))
            u = rn(z, model.w.final_norm)
            tok = int((W @ u).argmax())
            assert tok == out.tokens[b][k]
            a = u


def test_draft_chain_follows_the_diagonal():
    """Successor construction: identity block, P passing only the embedding half, and W_lm row
    sigma(t) aligned with N_e(E[t]).  The head then predicts x_{p+2} = sigma(x_{p+1}) from the
    token embedding it is given, so the chain drafted after pending token y must be
    sigma(y), sigma^2(y), sigma^3(y): depth k uses e = E(x^_{k-1}) at row p = j+k-1."""
    sh = TINY.replace(vocab=30, hidden=64, n_heads=2, head_dim=8)
    model = tiny_model(9, shape=sh, std=0.3, gain_std=0.0)
    dr = _tiny_drafter(9, model, gain_std=0.0)
    dr.dw.wo = torch.zeros_like(dr.dw.wo)
    dr.dw.w_down = torch.zeros_like(dr.dw.w_down)
    d = sh.hidden
    dr.dw.eh_proj = torch.cat([torch.eye(d), torch.zeros(d, d)], 1).to(torch.bfloat16)
    sigma = np.random.default_rng(1).permutation(sh.vocab)
    E = model.w.embed.to(F64)
    en = E / E.pow(2).mean(-1, keepdim=True).sqrt()
    W = torch.zeros(sh.vocab, d, dtype=F64)
    for t in range(sh.vocab):
        W[sigma[t]] = en[t]
    model.w.lm_head = W.to(torch.bfloat16)
    model._lm = None
    caches = tiny_caches(sh, 9, 3, 2, 5)
    dcs = _dcaches(sh, caches, 9)
    vo = O.verify(model, caches, [[c.pending] for c in caches], rb=False)
    O.commit(caches, vo, [[c.pending] for c in caches], dcs)
    out = O.draft(dr, dcs, 3, rb=False)
    for b, c in enumerate(caches):
        y = c.pending
        assert out.tokens[b] == [int(sigma[y]), int(sigma[sigma[y]]), int(sigma[sigma[sigma[y]]])]


def test_deep_draft_depths_attend_to_tentative_rows():
    """Closed form in which the draft block's attention matters at every depth: W_k = 0 and a
    zero key prefix make every score 0, so attention is the plain mean of the value rows the
    query may see; W_down = 0 makes the FFN add nothing.  Depth k at row p = j + k - 1 must see
    the committed rows 0..j, the tentative rows j+1..p-1 written by the shallower depths of the
    same chain, and its own row p (Sec. 3.1, Fig. "FastMTP state-shift alignment").  The chain is
    recomputed here with library primitives only and compared state by state; a chain that
    dropped the tentative rows is shown to differ."""
    model = tiny_model(14)
    dr = _tiny_drafter(14, model)
    H, hd, d = TINY.n_heads, TINY.head_dim, TINY.hidden
    wqkv = dr.dw.wqkv.clone()
    wqkv[H * hd:2 * H * hd] = 0
    dr.dw.wqkv = wqkv
    dr.dw.w_down = torch.zeros_like(dr.dw.w_down)
    caches = tiny_caches(TINY, 14, 2, 4, 7)
    dcs = []
    for b, c in enumerate(caches):
        kv = S.draft_kv_prefix(14, b, c.ctx, H, hd).clone()
        kv[0] = 0                                     # committed keys: zero
        dcs.append(O.DraftCache.from_prefix(kv))
    vprefix = [dc.v.clone() for dc in dcs]
    vo = O.verify(model, caches, [[c.pending] for c in caches], rb=False)
    O.commit(caches, vo, [[c.pending] for c in caches], dcs)
    rows_b = [dc.rows_b.clone() for dc in dcs]
    rows_t = [list(dc.rows_tok) for dc in dcs]
    K = 4
    out = O.draft(dr, dcs, K, rb=False)

    eps = TINY.rms_eps
    rn = lambda x, g: F.rms_norm(x, (d,), g.to(F64), eps=eps)
    E, W = model.w.embed.to(F64), model.w.lm_head.to(F64)
    Pm, Wv, Wo = dr.dw.eh_proj.to(F64), dr.dw.wqkv.to(F64)[2 * H * hd:], dr.dw.wo.to(F64)

    def z_of(tok, a):
        return F.linear(torch.cat([rn(E[tok], dr.dw.enorm), rn(a, dr.dw.hnorm)]), Pm)

    def v_of(z):
        return F.linear(rn(z, dr.dw.attn_norm), Wv)

    for b in range(2):
        vrows = list(vprefix[b].reshape(-1, H * hd))
        for a, tok in zip(rows_b[b], rows_t[b]):      # committed rows keep their base states
            z = z_of(tok, a.to(F64))
            vrows.append(v_of(z))
        n_committed = len(vrows)
        u_alt = None
        for k in range(K):
            if k > 0:
                z = z_of(tok, u)
                vrows.append(v_of(z))                 # row p of depth k+1 (tentative)
            mean_v = torch.stack(vrows).mean(0)       # uniform weights over rows 0..p
            u = rn(z + F.linear(mean_v, Wo), model.w.final_norm)
            assert torch.allclose(out.u[b][k], u, atol=1e-10, rtol=0), (b, k)
            if k == 2:
                # the same depth without the tentative row of depth 2: must be different
                seen = vrows[:n_committed] + vrows[-1:]
                u_alt = rn(z + F.linear(torch.stack(seen).mean(0), Wo), model.w.final_norm)
            tok = int(F.linear(u, W).argmax())
            assert tok == out.tokens[b][k], (b, k)
        assert not torch.allclose(u_alt, out.u[b][2], atol=1e-6)


def test_draft_cache_tracks_committed_length_and_base_states():
    """After every draft step the draft cache holds exactly the committed rows (same length as
    the verifier cache), and the committed rows' K/V come from the base states b_p."""
    model = tiny_model(10, std=0.5)
    dr = _tiny_drafter(10, model)
    caches = tiny_caches(TINY, 10, 2, 3, 7)
    dcs = _dcaches(TINY, caches, 10)
    vo = O.verify(model, caches, [[c.pending] for c in caches], rb=True)
    O.commit(caches, vo, [[c.pending] for c in caches], dcs)
    for _ in range(4):
        rows = [(dc.rows_b.clone(), list(dc.rows_tok), dc.ctx) for dc in dcs]
        drafts = O.draft(dr, dcs, 3, rb=True)
        for b, dc in enumerate(dcs):
            assert dc.ctx == caches[b].ctx
            rb_, rt, c0 = rows[b]
            z = O.model._draft_input(dr, rt, rb_, True)
            k, v = O.model._draft_kv_rows(dr, z, range(c0, c0 + len(rt)), True)
            assert torch.equal(dc.k[c0:], k) and torch.equal(dc.v[c0:], v)
        cand = [[c.pending] + drafts.tokens[b] for b, c in enumerate(caches)]
        vo = O.verify(model, caches, cand, rb=True)
        O.commit(caches, vo, cand, dcs)


def test_speculative_with_draft_head_equals_greedy():
    model = tiny_model(11, std=0.5)
    dr = _tiny_drafter(11, model)
    base = tiny_caches(TINY.replace(), 11, 2, 3, 6)
    greedy = O.greedy_decode(model, _clone(base), 10, rb=True)
    dcs = _dcaches(TINY, base, 11)
    st = O.DecodeStats()
    got = O.speculative_decode(model, _clone(base), 10, 3, drafter=dr, dcaches=dcs, rb=True, stats=st)
    assert got == greedy
    assert st.steps > 0


def test_lossless_with_accepting_draft_head():
    """Successor-map weights make the FastMTP head agree with the verifier often; the committed
    stream must still equal plain greedy decoding, now with long accepted prefixes."""
    sh = TINY.replace(hidden=64, n_heads=2, head_dim=8, vocab=60, n_layers=2)
    vw, dw, pi = S.successor_weights(sh, 13, 1.0, gain_std=0.0)
    model = O.Verifier(vw)
    dr = O.Drafter(dw, model)
    base = tiny_caches(sh, 13, 2, 3, 6)
    greedy = O.greedy_decode(model, _clone(base), 16, rb=True)
    assert greedy[0][:3] == [int(pi[base[0].pending]), int(pi[pi[base[0].pending]]),
                             int(pi[pi[pi[base[0].pending]]])]      # the verifier follows pi
    dcs = _dcaches(sh, base, 13)
    st = O.DecodeStats()
    got = O.speculative_decode(model, _clone(base), 16, 3, drafter=dr, dcaches=dcs, rb=True, stats=st)
    assert got == greedy
    assert sum(st.accept_hist[1:]) > 0


# ----------------------------------------------------------------------------- paper numbers

def test_shape_contract_parameter_counts_match_paper():
    spec = json.load(open(os.path.join(GOLD, "paper_model_spec.json")))
    s = S.ModelShape()
    assert (s.n_layers, s.hidden, s.n_experts, s.n_shared, s.top_k, s.vocab) == (
        spec["decoder_layers"], spec["hidden"], spec["routed_experts"], spec["shared_experts"],
        spec["top_k"], spec["vocab"])
    assert s.rope_theta == spec["rope_theta"] and s.max_position == spec["position_limit"]
    d, H, hd, E, I = s.hidden, s.n_heads, s.head_dim, s.n_experts, s.expert_inter
    attn = 3 * H * hd * d + d * H * hd
    expert = 3 * d * I
    per_layer_active = attn + E * d + (s.top_k + s.n_shared) * expert
    per_layer_total = attn + E * d + (E + s.n_shared) * expert
    active = s.n_layers * per_layer_active + s.vocab * d
    total = s.n_layers * per_layer_total + 2 * s.vocab * d
    assert abs(active / spec["active_params_decoder_approx"] - 1) < 0.03     # ~570M
    assert abs(total / spec["total_params_decoder_approx"] - 1) < 0.06       # ~3B
