"""The fp8-expert variant (no counterpart in the paper: expert matrices as e4m3 codes with one fp32
scale per output row, e4m3 expert inputs and SwiGLU activations, tcgen05 kind::f8f6f4 products)
against the fp64 oracle's fp8 mode, which dequantises the same codes exactly and rounds the same
two tensors to e4m3.

Parity rule of the variant:
* identical expert inputs (layer 0 with W_o = 0, so the MoE sees the embedding rows on both
  sides): the layer's residual output within 1e-5 relative per row and the routing exact -- the
  expert products, scales, e4m3 writes and the gate/up -> down hand-off are exact up to fp32
  accumulation;
* end to end: within 6e-2 relative (b, the residual stream, committed K/V, router
  probabilities), routing and tokens exact above the margins.  e4m3 keeps 3 mantissa bits, so
  an input element lying within the upstream difference (fp32 vs fp64 attention and softmax,
  bf16 rounding decisions: ~1e-4 relative) of a rounding boundary moves by a whole step, 12.5 %
  of itself; one such step in one of an expert's 1280 inputs changes its gate/up products by
  about 0.125 / sqrt(1280) = 0.35 %, which moves ~2.8 % of the 896 e4m3 activations a step and
  the expert's output by about sqrt(25) x 0.125 / sqrt(896) = 2 %; three such events on a row
  give 6e-2 (the bf16 path rounds its activations to bf16, 2^-8, and keeps 2e-2);
* losslessness (speculative == greedy) and batch invariance exactly, GPU against GPU."""
import numpy as np
import pytest
import torch

import oracle as O
import synth_inputs as S
from paper_2609_03181_gb300 import fastmtp as F
from tests.gpu_util import rel_err, seq_prefixes
from tests.test_gpu_verify import run_verify_case

pytestmark = pytest.mark.gpu

FP8_TOL = 6e-2


@pytest.mark.parametrize("B", [1, 8, 160])
def test_fp8_experts_exact_on_identical_inputs(B):
    """T = 4, 32 and 640 rows (the last with 128-row dual expert items)."""
    shape = S.ModelShape(n_layers=1, vocab=4096)
    seed = 21
    vw = S.verifier_weights(shape, seed, gain_std=0.1)
    vw.layers[0].wo = torch.zeros_like(vw.layers[0].wo)
    vw = S.quantize_experts_fp8(vw)
    dw = S.draft_weights(shape, seed)
    ctx = [20 + (7 * b) % 90 for b in range(B)]
    kvs, dkvs = seq_prefixes(shape, seed, ctx)
    pend = [int(t) for t in S.integers(seed, "pending", B, 0, shape.vocab - 1)]
    cand = [[pend[b], 5, 6, 7] for b in range(B)]
    ref = O.verify(O.Verifier(vw), [O.SeqCache.from_prefix(kvs[b], pend[b]) for b in range(B)], cand, rb=True,
                   keep_hidden=True)
    eng = F.Engine(vw, dw, max_batch=B, K_max=3, max_ctx=max(ctx) + 8, page_size=64, expert_fp8=True)
    for b in range(B):
        eng.load_prefix(b, kvs[b], dkvs[b], pend[b])
    dev = torch.device("cuda")
    vt = torch.empty(B, 4, dtype=torch.int32, device=dev)
    acc = torch.empty(B, dtype=torch.int32, device=dev)
    eng.verify_step(torch.arange(B, dtype=torch.int32, device=dev), torch.tensor(cand, dtype=torch.int32, device=dev),
                    vt, acc)
    eng.sync()
    T = 4 * B
    h = eng.read_workspace(F.WS_HIDDEN, (T, shape.hidden), torch.float32)
    ridx = eng.read_workspace(F.WS_ROUTE_IDX, (1, eng.max_batch * 4, 6), torch.int32)[0, :T].numpy()
    eng.close()
    same = (np.sort(ridx, -1) == np.sort(ref.route_idx[0].numpy(), -1)).all(-1)
    gaps = ref.route_gap[0].numpy()
    assert same[gaps > 1e-3].all()
    errs = [rel_err(h[i], ref.hidden[-1][i]) for i in range(T) if same[i]]
    print(f"[parity] fp8 experts, identical inputs, T={T}: max residual rel err {max(errs):.3g}")
    assert max(errs) < 1e-5


def test_fp8_verify_one_layer_b1_ctx512():
    run_verify_case(S.ModelShape(n_layers=1), 0, [512], K=3, fp8=True, rel_tol=FP8_TOL)


def test_fp8_verify_two_layers_ragged_contexts():
    run_verify_case(S.ModelShape(n_layers=2, vocab=4096), 5, [0, 1, 63, 64, 129, 200], K=2, fp8=True,
                    rel_tol=FP8_TOL)


def test_fp8_verify_batch_256_large_tiles():
    """T = 1024 candidate rows: the expert launch runs 128-row dual items on e4m3 operands."""
    ctx = [int(c) for c in S.integers(9, "ctx", 256, 1, 160)]
    run_verify_case(S.ModelShape(n_layers=1, vocab=4096), 9, ctx, K=3, check=range(3, 256, 16), fp8=True,
                    rel_tol=FP8_TOL)


def _loop(eng, B, K, n_tok, drafts=None):
    dev = torch.device("cuda")
    slots = torch.arange(B, dtype=torch.int32, device=dev)
    out = [[] for _ in range(B)]
    while min(len(o) for o in out) < n_tok:
        pend = [eng.seq_state(b)[1] for b in range(B)]
        cand = torch.tensor([[pend[b]] + (drafts(b, out[b]) if drafts else []) for b in range(B)],
                            dtype=torch.int32, device=dev)
        Kc = cand.shape[1] - 1
        vt = torch.empty(B, Kc + 1, dtype=torch.int32, device=dev)
        acc = torch.empty(B, dtype=torch.int32, device=dev)
        eng.verify_step(slots, cand, vt, acc)
        com = torch.empty(B, Kc + 1, dtype=torch.int32, device=dev)
        nc = torch.empty(B, dtype=torch.int32, device=dev)
        eng.accept_commit(slots, com, nc)
        eng.sync()
        for b in range(B):
            out[b].extend(com[b, : int(nc[b])].tolist())
    return [o[:n_tok] for o in out]


def test_fp8_speculative_equals_greedy_and_batch_invariance():
    shape = S.ModelShape(n_layers=2, vocab=4096)
    seed, B, K, n = 41, 4, 3, 16
    vw = S.quantize_experts_fp8(S.verifier_weights(shape, seed, gain_std=0.1))
    dw = S.draft_weights(shape, seed, gain_std=0.1)
    Bb = 128
    ctx = [int(c) for c in S.integers(seed, "ctx", Bb, 30, 200)]
    kvs = [S.kv_prefix(seed, b, shape.n_layers, ctx[b], shape.n_heads, shape.head_dim) for b in range(Bb)]
    dkvs = [S.draft_kv_prefix(seed, b, ctx[b], shape.n_heads, shape.head_dim) for b in range(Bb)]
    pend = [int(x) for x in S.integers(seed, "pending", Bb, 0, shape.vocab - 1)]
    eng = F.Engine(vw, dw, max_batch=Bb, K_max=K, max_ctx=max(ctx) + 2 * n + 16, page_size=64, expert_fp8=True)

    def reset(nb):
        for b in range(nb):
            eng.load_prefix(b, kvs[b], dkvs[b], pend[b])

    reset(B)
    greedy = _loop(eng, B, 0, n + K + 2)
    for name, fn in (("right", lambda b, done: greedy[b][len(done):len(done) + K]),
                     ("wrong", lambda b, done: [(t + 1) % shape.vocab for t in greedy[b][len(done):len(done) + K]])):
        reset(B)
        assert _loop(eng, B, K, n, fn) == [g[:n] for g in greedy], name
    # sequence 0 alone, in a batch of 4 (16 rows) and in a batch of 128 (512 rows: 128-row dual expert
    # tiles): bit-identical b rows and verifier tokens
    dev = torch.device("cuda")
    res = []
    for bsz in (1, B, Bb):
        reset(bsz)
        slots = torch.arange(bsz, dtype=torch.int32, device=dev)
        cand = torch.tensor([[pend[b], 11, 12, 13] for b in range(bsz)], dtype=torch.int32, device=dev)
        vt = torch.empty(bsz, K + 1, dtype=torch.int32, device=dev)
        acc = torch.empty(bsz, dtype=torch.int32, device=dev)
        eng.verify_step(slots, cand, vt, acc)
        bst = eng.read_workspace(F.WS_B, (bsz * (K + 1), shape.hidden), torch.bfloat16)
        com = torch.empty(bsz, K + 1, dtype=torch.int32, device=dev)
        nc = torch.empty(bsz, dtype=torch.int32, device=dev)
        eng.accept_commit(slots, com, nc)
        eng.sync()
        res.append((bst[: K + 1].clone(), vt[0].cpu().clone()))
    eng.close()
    for other in res[1:]:
        assert torch.equal(res[0][0], other[0]) and torch.equal(res[0][1], other[1])
