"""Seeded synthetic inputs for the FastMTP speculative decode step.

This module only draws random numbers: the shape contract of the compact MoE decoder
(Table "Model specification": 12 layers, d=1280, 64 routed + 2 shared experts, top-6,
vocabulary 129,280, RoPE theta 1e6, position limit 32,768) with the shapes the paper leaves
open (10 heads x 128, expert intermediate 896, draft-block intermediate 3584, RMSNorm eps
1e-6), random bf16 weights ~N(0, 0.02), synthetic committed KV prefixes ~N(0, 1), context
lengths, token ids and coin flips.  It holds none of the method's arithmetic, so both the
fp64 oracle and the CUDA path can take their inputs from it without sharing any compute code.

Every tensor is drawn from its own Philox stream keyed by (seed, name, chunk), so any single
tensor (one expert's matrices, one sequence's KV prefix) can be regenerated on its own and
large tensors are filled by several threads at once.
"""
from __future__ import annotations

import math
import zlib
from concurrent.futures import ThreadPoolExecutor
from dataclasses import dataclass, field
from typing import List, Optional

import numpy as np
import torch

_CHUNK = 1 << 22  # elements per Philox stream


@dataclass(frozen=True)
class ModelShape:
    hidden: int = 1280
    n_heads: int = 10
    head_dim: int = 128
    n_layers: int = 12
    n_experts: int = 64
    top_k: int = 6
    n_shared: int = 2
    expert_inter: int = 896
    draft_inter: int = 3584
    vocab: int = 129280
    rms_eps: float = 1e-6
    rope_theta: float = 1.0e6
    max_position: int = 32768

    def replace(self, **kw) -> "ModelShape":
        d = dict(self.__dict__)
        d.update(kw)
        return ModelShape(**d)


@dataclass(frozen=True)
class Workload:
    """One of the five workloads of the verify/draft step: sizes, seeds and the input recipe
    only.  ctx is the committed context range U[ctx_lo, ctx_hi] per sequence (the first
    `visual` positions stand in for the page's visual tokens); `draft_only` runs the draft block
    alone; `gen_tokens` is the number of committed tokens a loop workload generates; `grid`
    holds the sweep's axes."""
    name: str
    n_layers: int
    batch: int
    K: int
    ctx_lo: int
    ctx_hi: int
    seed: int
    visual: int = 0
    p_match: float = 0.0
    draft_only: bool = False
    gen_tokens: int = 0
    grid: Optional[dict] = None


# The five workloads of the verify/draft step (seeded, synthetic), named by what they are.
WORKLOADS = {
    "one_layer_b1_ctx512": Workload("one decoder layer, verify step", n_layers=1, batch=1, K=3, ctx_lo=512, ctx_hi=512,
                     seed=0, p_match=0.7),
    "verify_12l_b8_ctx768_1024": Workload("12-layer verifier, verify step", n_layers=12, batch=8, K=3, ctx_lo=768, ctx_hi=1024,
                     seed=1, visual=256),
    "draft_block_b32_ctx2048": Workload("draft block alone", n_layers=0, batch=32, K=3, ctx_lo=2048, ctx_hi=2048, seed=2,
                     draft_only=True),
    "loop_12l_b64_ctx1024_4096": Workload("speculative decode loop, verifier + draft block", n_layers=12, batch=64, K=3,
                     ctx_lo=1024, ctx_hi=4096, seed=3, gen_tokens=512),
    "sweep_12l_b1_256_ctx1024_8192": Workload("verify-throughput sweep", n_layers=12, batch=256, K=3, ctx_lo=1024, ctx_hi=8192, seed=4,
                     grid={"batch": (1, 4, 16, 64, 256), "ctx": (1024, 4096, 8192), "K": (0, 1, 2, 3),
                           "router": ("uniform", "zipf"), "zipf_s": 1.2, "seeds": (4, 5, 6, 7, 8)}),
}


def _stream(seed: int, name: str, chunk: int) -> np.random.Generator:
    ss = np.random.SeedSequence([int(seed) & 0xFFFFFFFF, zlib.crc32(name.encode()), int(chunk)])
    return np.random.Generator(np.random.Philox(ss))


_POOL: Optional[ThreadPoolExecutor] = None


def _pool() -> ThreadPoolExecutor:
    global _POOL
    if _POOL is None:
        import os
        _POOL = ThreadPoolExecutor(max_workers=max(1, min(32, os.cpu_count() or 1)))
    return _POOL


def normal(seed: int, name: str, shape, std: float = 1.0, dtype=torch.bfloat16) -> torch.Tensor:
    """N(0, std^2) samples of the given shape, rounded to `dtype` (bf16 by default)."""
    n = int(np.prod(shape)) if len(shape) else 1
    out = np.empty(n, dtype=np.float32)
    nchunks = (n + _CHUNK - 1) // _CHUNK

    def fill(c):
        lo, hi = c * _CHUNK, min(n, (c + 1) * _CHUNK)
        g = _stream(seed, name, c)
        g.standard_normal(hi - lo, dtype=np.float32, out=out[lo:hi])
        if std != 1.0:
            out[lo:hi] *= np.float32(std)

    if nchunks > 1:
        list(_pool().map(fill, range(nchunks)))
    elif n:
        fill(0)
    return torch.from_numpy(out).reshape(tuple(shape)).to(dtype)


def integers(seed: int, name: str, n: int, lo: int, hi: int) -> np.ndarray:
    """n integers uniform in [lo, hi] (inclusive), int64."""
    return _stream(seed, name, 0).integers(lo, hi + 1, size=n, dtype=np.int64)


def uniforms(seed: int, name: str, n: int) -> np.ndarray:
    """n floats uniform in [0, 1), float64."""
    return _stream(seed, name, 0).random(n)


def permutation(seed: int, name: str, n: int) -> np.ndarray:
    return _stream(seed, name, 0).permutation(n)


def _gain(seed: int, name: str, d: int, gain_std: float) -> torch.Tensor:
    """RMSNorm gain: exactly 1 (the workloads' initialisation) or 1 + N(0, gain_std^2)."""
    if gain_std == 0.0:
        return torch.ones(d, dtype=torch.bfloat16)
    return (1.0 + normal(seed, name, (d,), gain_std, torch.float32)).to(torch.bfloat16)


@dataclass
class LayerWeights:
    attn_norm: torch.Tensor        # [d]
    wqkv: torch.Tensor             # [3d][d]  rows: q (H*hd), k (H*hd), v (H*hd)
    wo: torch.Tensor               # [d][H*hd]
    moe_norm: torch.Tensor         # [d]
    router: torch.Tensor           # [E][d]
    w_gate_up: torch.Tensor        # [E][2I][d]  rows 0..I-1 gate, I..2I-1 up
    w_down: torch.Tensor           # [E][d][I]
    shared_gate_up: torch.Tensor   # [S][2I][d]
    shared_down: torch.Tensor      # [S][d][I]
    router_bias: Optional[torch.Tensor] = None  # fp32 [E] or None


@dataclass
class VerifierWeights:
    shape: ModelShape
    embed: torch.Tensor        # [V][d]
    lm_head: torch.Tensor      # [V][d]
    final_norm: torch.Tensor   # [d]
    layers: List[LayerWeights] = field(default_factory=list)


@dataclass
class DraftWeights:
    enorm: torch.Tensor        # [d]
    hnorm: torch.Tensor        # [d]
    eh_proj: torch.Tensor      # [d][2d]  input = [N_e(e); N_h(a)]
    attn_norm: torch.Tensor    # [d]
    wqkv: torch.Tensor         # [3d][d]
    wo: torch.Tensor           # [d][d]
    ffn_norm: torch.Tensor     # [d]
    w_gate_up: torch.Tensor    # [2*Id][d] rows 0..Id-1 gate, Id..2Id-1 up
    w_down: torch.Tensor       # [d][Id]


def zipf_router_bias(seed: int, layer: int, n_experts: int, s: float = 1.2) -> torch.Tensor:
    """Per-expert router-logit bias -s*ln(rank) over a seeded permutation of the experts.

    Added to the router logits it makes P(select expert of rank r) fall off like r^-s, the
    skewed-load case of the throughput sweep."""
    rank = permutation(seed, f"zipf.{layer}", n_experts) + 1
    return torch.tensor([-s * math.log(r) for r in rank], dtype=torch.float32)


def verifier_weights(shape: ModelShape, seed: int, std: float = 0.02, gain_std: float = 0.0,
                     zipf_s: Optional[float] = None) -> VerifierWeights:
    d, H, hd, E, I, S = (shape.hidden, shape.n_heads, shape.head_dim, shape.n_experts,
                         shape.expert_inter, shape.n_shared)
    w = VerifierWeights(
        shape=shape,
        embed=normal(seed, "embed", (shape.vocab, d), std),
        lm_head=normal(seed, "lm_head", (shape.vocab, d), std),
        final_norm=_gain(seed, "final_norm", d, gain_std),
    )
    for l in range(shape.n_layers):
        w.layers.append(LayerWeights(
            attn_norm=_gain(seed, f"l{l}.attn_norm", d, gain_std),
            wqkv=normal(seed, f"l{l}.wqkv", (3 * H * hd, d), std),
            wo=normal(seed, f"l{l}.wo", (d, H * hd), std),
            moe_norm=_gain(seed, f"l{l}.moe_norm", d, gain_std),
            router=normal(seed, f"l{l}.router", (E, d), std),
            w_gate_up=normal(seed, f"l{l}.w_gate_up", (E, 2 * I, d), std),
            w_down=normal(seed, f"l{l}.w_down", (E, d, I), std),
            shared_gate_up=normal(seed, f"l{l}.shared_gate_up", (S, 2 * I, d), std),
            shared_down=normal(seed, f"l{l}.shared_down", (S, d, I), std),
            router_bias=(zipf_router_bias(seed, l, E, zipf_s) if zipf_s else None),
        ))
    return w


def draft_weights(shape: ModelShape, seed: int, std: float = 0.02, gain_std: float = 0.0) -> DraftWeights:
    d, H, hd, Id = shape.hidden, shape.n_heads, shape.head_dim, shape.draft_inter
    return DraftWeights(
        enorm=_gain(seed, "mtp.enorm", d, gain_std),
        hnorm=_gain(seed, "mtp.hnorm", d, gain_std),
        eh_proj=normal(seed, "mtp.eh_proj", (d, 2 * d), std),
        attn_norm=_gain(seed, "mtp.attn_norm", d, gain_std),
        wqkv=normal(seed, "mtp.wqkv", (3 * H * hd, d), std),
        wo=normal(seed, "mtp.wo", (d, H * hd), std),
        ffn_norm=_gain(seed, "mtp.ffn_norm", d, gain_std),
        w_gate_up=normal(seed, "mtp.w_gate_up", (2 * Id, d), std),
        w_down=normal(seed, "mtp.w_down", (d, Id), std),
    )


def kv_prefix(seed: int, seq: int, n_layers: int, ctx: int, n_heads: int, head_dim: int) -> torch.Tensor:
    """Committed verifier KV for positions 0..ctx-1 of one sequence, bf16 [L][2][ctx][H][hd] ~N(0,1).

    It stands in for the prefill of the 256 + 100n visual tokens and the prompt; keys are taken
    as already rotated (the cache stores post-RoPE keys)."""
    return normal(seed, f"kv.{seq}", (n_layers, 2, ctx, n_heads, head_dim), 1.0)


def draft_kv_prefix(seed: int, seq: int, ctx: int, n_heads: int, head_dim: int) -> torch.Tensor:
    """Committed draft-block KV for rows 0..ctx-1 of one sequence, bf16 [2][ctx][H][hd] ~N(0,1)."""
    return normal(seed, f"dkv.{seq}", (2, ctx, n_heads, head_dim), 1.0)


def successor_weights(shape: ModelShape, seed: int, beta_over_alpha: float, alpha: float = 1.0,
                      std: float = 0.02, gain_std: float = 0.0):
    """Weights under which speculative decoding accepts a tunable share of the drafts.

    Input construction only (seeded random matrices, a permutation and scalings):
    * E ~ N(0, 1) (instead of 0.02) so the embedding dominates the residual stream of the
      random std-0.02 layers, and W_lm[v] = E[pi^-1(v)] for a seeded permutation pi of the
      vocabulary: the verifier's greedy successor of token x is pi(x), by a wide margin;
    * P = [alpha * I | beta * M] with M ~ N(0, 1/d): the draft head sees the next token's
      embedding through the identity half and a random rotation of its input state through the
      other half; the ratio beta/alpha sets how often that perturbation moves the draft's argmax
      away from pi(x), i.e. the acceptance rate.
    Returns (VerifierWeights, DraftWeights, pi)."""
    vw = verifier_weights(shape, seed, std=std, gain_std=gain_std)
    dw = draft_weights(shape, seed, std=std, gain_std=gain_std)
    d, V = shape.hidden, shape.vocab
    E = normal(seed, "succ.embed", (V, d), 1.0)
    pi = permutation(seed, "succ.pi", V)
    inv = np.empty(V, dtype=np.int64)
    inv[pi] = np.arange(V)
    vw.embed = E
    vw.lm_head = E[torch.from_numpy(inv)].contiguous()
    M = normal(seed, "succ.M", (d, d), 1.0 / math.sqrt(d), dtype=torch.float32)
    eye = torch.eye(d, dtype=torch.float32)
    dw.eh_proj = torch.cat([alpha * eye, (alpha * beta_over_alpha) * M], dim=1).to(torch.bfloat16).contiguous()
    return vw, dw, pi


def quantize_experts_fp8(vw: "VerifierWeights") -> "VerifierWeights":
    """The fp8-expert variant of a verifier (input construction only): every routed and shared
    expert matrix stored as e4m3 byte codes with one fp32 scale per output row, scale =
    max |row| / 448, codes = the row divided by its scale rounded to the nearest e4m3 value (ties
    to even, through PyTorch's float8_e4m3fn conversion).  Adds the fields w_gate_up_f8,
    gate_up_scale, w_down_f8, down_scale, shared_gate_up_f8, shared_gate_up_scale,
    shared_down_f8, shared_down_scale (uint8 codes, fp32 scales) to a copy of every layer; the
    bf16 matrices stay as they were."""
    import copy

    def q(w):
        wf = w.float()
        sc = wf.abs().amax(-1).clamp_min(1e-30) / 448.0
        codes = (wf / sc[..., None]).clamp(-448.0, 448.0).to(torch.float8_e4m3fn).view(torch.uint8)
        return codes.contiguous(), sc.contiguous()

    out = copy.copy(vw)
    out.layers = []
    for lw in vw.layers:
        l2 = copy.copy(lw)
        l2.w_gate_up_f8, l2.gate_up_scale = q(lw.w_gate_up)
        l2.w_down_f8, l2.down_scale = q(lw.w_down)
        l2.shared_gate_up_f8, l2.shared_gate_up_scale = q(lw.shared_gate_up)
        l2.shared_down_f8, l2.shared_down_scale = q(lw.shared_down)
        out.layers.append(l2)
    return out


def kv_prefix_device(seed: int, seq: int, n_layers: int, ctx: int, n_heads: int, head_dim: int,
                     device) -> torch.Tensor:
    """Like kv_prefix, drawn on `device` by PyTorch's seeded generator (a different stream from
    kv_prefix's): for large GPU-only workloads whose prefixes no CPU oracle has to reproduce."""
    g = torch.Generator(device=device)
    g.manual_seed((int(seed) * 1000003 + zlib.crc32(f"kvdev.{seq}".encode())) & 0x7FFFFFFFFFFFFFFF)
    x = torch.randn(n_layers, 2, ctx, n_heads, head_dim, generator=g, device=device, dtype=torch.float32)
    return x.to(torch.bfloat16)


def draft_kv_prefix_device(seed: int, seq: int, ctx: int, n_heads: int, head_dim: int, device) -> torch.Tensor:
    g = torch.Generator(device=device)
    g.manual_seed((int(seed) * 1000003 + zlib.crc32(f"dkvdev.{seq}".encode())) & 0x7FFFFFFFFFFFFFFF)
    return torch.randn(2, ctx, n_heads, head_dim, generator=g, device=device, dtype=torch.float32).to(torch.bfloat16)
