"""End-to-end speculative greedy decoding at serving scale: the 12-layer MoE
verifier plus the FastMTP draft block, batch 64, prompt contexts U[1024, 4096], 512 generated
tokens per sequence, acceptance-tuned weights (successor map, beta/alpha = 7).  The committed
streams must equal plain greedy decoding token for token (Sec. 3.1: lossless), with drafts
actually accepted.  GPU only: speculative GPU vs greedy GPU (the prefixes are drawn on the
device; no oracle copy is needed)."""
import numpy as np
import pytest
import torch

import synth_inputs as S
from paper_2609_03181_gb300 import fastmtp as F

pytestmark = pytest.mark.gpu

B, K, N_TOK, SEED = 64, 3, 512, 3


def decode(eng, slots, pend, K_step):
    """Runs the loop on the engine's stream; returns [B][N_TOK] committed tokens and the accept
    lengths of the speculative steps."""
    dev = slots.device
    s = eng.stream
    hist_tok, hist_n, ms = [], [], []
    with torch.cuda.stream(s):
        cand0 = torch.tensor([[p] for p in pend], dtype=torch.int32, device=dev)
        com0 = torch.empty(B, 1, dtype=torch.int32, device=dev)
        acc = torch.empty(B, dtype=torch.int32, device=dev)
        n0 = torch.empty(B, dtype=torch.int32, device=dev)
        v0 = torch.empty(B, 1, dtype=torch.int32, device=dev)
        cand = torch.empty(B, K + 1, dtype=torch.int32, device=dev)
        vt = torch.empty(B, K + 1, dtype=torch.int32, device=dev)
        com = torch.empty(B, K + 1, dtype=torch.int32, device=dev)
        ncom = torch.empty(B, dtype=torch.int32, device=dev)
    s.synchronize()
    total = np.zeros(B, dtype=np.int64)
    step = 0
    while total.min() < N_TOK:
        for _ in range(16):
            if K_step == 0 or step == 0:
                eng.verify_step(slots, cand0, v0, acc)
                eng.accept_commit(slots, com0, n0)
                with torch.cuda.stream(s):
                    cand0.copy_(com0)          # the committed token is the next pending token
                    hist_tok.append(torch.nn.functional.pad(com0, (0, K)).clone())
                    hist_n.append(n0.clone())
            else:
                eng.draft_step(slots, K, cand)
                eng.verify_step(slots, cand, vt, acc)
                eng.accept_commit(slots, com, ncom)
                with torch.cuda.stream(s):
                    hist_tok.append(com.clone())
                    hist_n.append(ncom.clone())
                    ms.append(acc.clone())
            step += 1
        eng.sync()
        total = torch.stack(hist_n).sum(0).cpu().numpy()
    toks = torch.stack(hist_tok).cpu().numpy()
    ns = torch.stack(hist_n).cpu().numpy()
    out = []
    for b in range(B):
        seq = []
        for i in range(len(ns)):
            seq.extend(toks[i, b, :ns[i, b]].tolist())
        out.append(seq[:N_TOK])
    return out, (torch.stack(ms).cpu().numpy() if ms else np.zeros(0))


def test_speculative_equals_greedy_b64_512_tokens():
    shape = S.ModelShape()
    vw, dw, _ = S.successor_weights(shape, SEED, 7.0)
    ctx = [int(c) for c in S.integers(SEED, "ctx", B, 1024, 4096)]
    pend = [int(t) for t in S.integers(SEED, "pending", B, 0, shape.vocab - 1)]
    eng = F.Engine(vw, dw, max_batch=B, K_max=K, max_ctx=max(ctx) + N_TOK + 4 * (K + 1) + 16, page_size=64)
    dev = torch.device("cuda")
    slots = torch.arange(B, dtype=torch.int32, device=dev)

    def reset():
        for b in range(B):
            kv = S.kv_prefix_device(SEED, b, shape.n_layers, ctx[b], shape.n_heads, shape.head_dim, dev)
            dkv = S.draft_kv_prefix_device(SEED, b, ctx[b], shape.n_heads, shape.head_dim, dev)
            eng.load_prefix(b, kv, dkv, pend[b])

    reset()
    greedy, _ = decode(eng, slots, pend, 0)
    reset()
    spec, ms = decode(eng, slots, pend, K)
    eng.close()
    for b in range(B):
        assert spec[b] == greedy[b], f"sequence {b} diverges at token {next(i for i in range(N_TOK) if spec[b][i] != greedy[b][i])}"
    tau = 1 + ms.mean()
    assert tau > 1.5, f"tau {tau}"
