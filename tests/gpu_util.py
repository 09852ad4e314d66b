"""Helpers of the GPU parity tests: seeded workloads, engines, and the comparison rules.

Comparison rules (written out in each test): floating-point tensors within a max relative
error max|gpu - ref| / max|ref| of 2e-2 (bf16 storage); indices (router experts, argmax tokens,
accept lengths) bit-exact wherever the fp64 oracle's top-2 margin exceeds 1e-3, counted and
skipped below it."""
import numpy as np
import torch

import oracle as O
import synth_inputs as S

REL_TOL = 2e-2
GAP = 1e-3


def rel_err(gpu, ref) -> float:
    gpu = gpu.double().cpu()
    ref = ref.double().cpu()
    return float((gpu - ref).abs().max() / ref.abs().max().clamp_min(1e-30))


def seq_prefixes(shape, seed, ctx_lens):
    kvs = [S.kv_prefix(seed, b, shape.n_layers, int(c), shape.n_heads, shape.head_dim) for b, c in enumerate(ctx_lens)]
    dkvs = [S.draft_kv_prefix(seed, b, int(c), shape.n_heads, shape.head_dim) for b, c in enumerate(ctx_lens)]
    return kvs, dkvs


def make_drafts(model, caches, K, seed, p_match=0.7, rb=True):
    """Draft tokens equal to the oracle's greedy token with probability p_match, else a uniform
    random id (drafts built one depth at a time, so accept lengths vary)."""
    B = len(caches)
    coins = S.uniforms(seed, "draft.coin", B * K).reshape(B, K)
    rand = S.integers(seed, "draft.tok", B * K, 0, model.s.vocab - 1).reshape(B, K)
    drafts = [[] for _ in range(B)]
    for r in range(K):
        cand = [[c.pending] + drafts[b] for b, c in enumerate(caches)]
        out = O.verify(model, caches, cand, rb=rb)
        for b in range(B):
            v = int(out.v[b, r])
            drafts[b].append(v if coins[b, r] < p_match else int(rand[b, r]))
    return [[c.pending] + drafts[b] for b, c in enumerate(caches)]


def index_parity(gpu_idx, ref_idx, gaps, gap=GAP):
    """Returns (n_checked, n_skipped, n_mismatch) over rows whose oracle gap exceeds `gap`."""
    gpu_idx = np.asarray(gpu_idx)
    ref_idx = np.asarray(ref_idx)
    gaps = np.asarray(gaps)
    ok = gaps > gap
    mism = int(((gpu_idx != ref_idx).reshape(len(gaps), -1).any(-1) & ok).sum())
    return int(ok.sum()), int((~ok).sum()), mism


def argmax_margin(lm_head, b_gpu, b_ref, k_sigma=8.0, floor=GAP):
    """Per-row margin for comparing argmax tokens: the oracle's top-2 logit gap must exceed
    k_sigma standard deviations of the logit-difference noise that the measured state
    difference implies, sqrt(2) * rms(W_lm) * ||b_gpu - b_ref||_2 (and at least `floor`).
    Twelve bf16 layers leave ~1% state noise, so a fixed 1e-3 logit margin would flip by chance."""
    w_rms = float(lm_head.float().pow(2).mean().sqrt())
    d = (b_gpu.double().cpu() - b_ref.double().cpu()).reshape(b_ref.shape[0], -1)
    return np.maximum(floor, k_sigma * np.sqrt(2.0) * w_rms * d.norm(dim=-1).numpy())
