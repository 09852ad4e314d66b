"""Plain fp64 oracle of the FastMTP speculative decode step on the compact MoE decoder.

TEST INFRASTRUCTURE: imported only by tests/, __graft_entry__.smoke() and bench.py's
CPU-baseline leg.  Nothing in the product library imports, links or runs it.

What it computes, in the paper's order and notation (arXiv 2609.03181, "Jina-OCR-v1"):

* the verifier: the DeepSeekMoE decoder of Table "Model specification" (12 layers, d=1280,
  64 routed + 2 shared experts, top-6, RoPE theta=1e6), run over the K+1 candidate tokens
  [bonus, x^_1..x^_K] of each sequence against its committed KV cache (Sec. 3, "Model
  Architecture"; the router notation p_{i,t} of Sec. 5.4 "Auxiliary regularizers");
* greedy verification: v_r = argmax q_r, the longest equality prefix m of the acceptance
  equation of Sec. 3.1, commit x^_{1:m} then v_{m+1} (bonus when m=K), discard the tail;
* the FastMTP draft head, the draft-head equation of Sec. 3.1: a^(1)_p = b_p,
  a^(k)_p = u^(k-1)_{p-1}, z = P([N_e(e_{p+1}); N_h(a)]), u = N_o(B_theta(z; pos=p)),
  l = W_lm u, with E, N_o and W_lm tied to the verifier, committed rows keeping their base
  states in the draft KV cache, and the inference chain on the diagonal p = j+k-1
  (Fig. "FastMTP state-shift alignment");
* plain greedy autoregressive decoding and the speculative loop built from the above.

Readings where the paper is silent (each also listed in the design notes): MHA 10x128 with
scale 1/sqrt(128); rotate-half RoPE over all 128 dims at the absolute position; pre-norm
layers, all 12 MoE; RMSNorm; router softmax over all experts, top-k by probability with ties
to the lower expert id, selected probabilities used as gates without renormalisation; shared
experts are SwiGLU experts of the routed width with gate 1; b_p = N_o(h_L); B_theta is a
pre-norm attention + SwiGLU block with its own KV cache; argmax ties go to the lower token id.

Precision: every quantity is fp64 computed from the bf16-stored weights and inputs.  With
`rb=True` ("storage rounding") values are additionally rounded to bf16, in one step and ties
to even, exactly where the GPU contract stores bf16 (norm outputs that feed a matrix product,
the rotated queries and K/V that feed the attention products, attention outputs, SwiGLU
activations, the states b and u); everything between those points stays fp64.  `rb=False` is
the plain definition.

fp8-expert variant (not in the paper; a precision option of this library): when a layer carries
e4m3 expert weights with one fp32 scale per output row (synth_inputs.quantize_experts_fp8), the
oracle dequantises them exactly (code value x scale, in fp64) and rounds the two tensors that enter
the expert products, the normalised input rows and the SwiGLU activations, to e4m3 (ties to even,
saturating at 448), where the bf16 path rounds the activations to bf16.

Parity of absolute hidden-state values on random weights is pinned only through the special
cases and invariants in tests/test_oracle_pins.py (closed forms, brute force, the identity
draft block, losslessness); beyond those the values are parity unpinned.
"""
from __future__ import annotations

import math
from dataclasses import dataclass, field
from typing import Callable, List, Optional, Sequence

import numpy as np
import torch

F64 = torch.float64

__all__ = [
    "round_bf16", "round_e4m3", "decode_e4m3", "dequant_rows", "rms_norm", "rope", "attention", "silu", "swiglu", "router_topk",
    "argmax_with_gap", "accept_length", "SeqCache", "DraftCache", "Verifier", "Drafter",
    "VerifyOut", "DraftOut", "verify", "commit", "draft", "greedy_decode",
    "speculative_decode", "DecodeStats",
]


# ----------------------------------------------------------------------------- precision

def round_bf16(x: torch.Tensor) -> torch.Tensor:
    """Round fp64 values to the nearest bfloat16 value (8 significant bits), ties to even.

    One rounding step straight from fp64 (not via fp32).  Values here never reach the bf16
    subnormal or overflow range; zeros stay zero."""
    a = x.detach().to(F64).contiguous().numpy()
    m, e = np.frexp(a)                     # a = m * 2**e with 0.5 <= |m| < 1
    r = np.rint(m * 256.0) / 256.0         # keep 8 significant bits; rint ties to even
    return torch.from_numpy(np.ldexp(r, e)).reshape(x.shape)


E4M3_MAX = 448.0


def round_e4m3(x: torch.Tensor) -> torch.Tensor:
    """Round to the nearest e4m3 value (1 sign, 4 exponent bits with bias 7, 3 mantissa bits, no
    infinities), ties to even, saturating: |x| >= 448 gives +-448.  Normal values keep 4
    significant bits (|x| >= 2^-6); below that the grid is the subnormal step 2^-9."""
    a = np.clip(x.detach().to(F64).contiguous().numpy(), -E4M3_MAX, E4M3_MAX)
    m, e = np.frexp(a)                                   # a = m * 2**e, 0.5 <= |m| < 1
    normal = np.ldexp(np.rint(m * 16.0) / 16.0, e)       # 4 significant bits, rint ties to even
    sub = np.rint(a / 2.0 ** -9) * 2.0 ** -9
    r = np.where(np.abs(a) >= 2.0 ** -6, normal, sub)
    return torch.from_numpy(np.clip(r, -E4M3_MAX, E4M3_MAX)).reshape(x.shape)


def decode_e4m3(codes: torch.Tensor) -> torch.Tensor:
    """Values of e4m3 byte codes (uint8): sign bit 7, exponent bits 6..3 (bias 7), mantissa bits
    2..0; exponent 0 is subnormal, m * 2^-9."""
    b = codes.to(torch.int64)
    s = torch.where((b >> 7) & 1 == 1, -1.0, 1.0).to(F64)
    e = (b >> 3) & 15
    m = (b & 7).to(F64)
    normal = (1.0 + m / 8.0) * torch.pow(torch.tensor(2.0, dtype=F64), (e - 7).to(F64))
    sub = m * 2.0 ** -9
    return s * torch.where(e == 0, sub, normal)


def dequant_rows(codes: torch.Tensor, scale: torch.Tensor) -> torch.Tensor:
    """fp8 weight matrix [.., rows, k] with one fp32 scale per row [.., rows]: values * scale."""
    return decode_e4m3(codes) * f64(scale)[..., None]


def _rb(x: torch.Tensor, on: bool) -> torch.Tensor:
    return round_bf16(x) if on else x


def f64(t: torch.Tensor) -> torch.Tensor:
    return t.to(F64)


# ----------------------------------------------------------------------------- primitives

def rms_norm(x: torch.Tensor, gain: torch.Tensor, eps: float) -> torch.Tensor:
    """RMSNorm over the last dim: x / sqrt(mean(x^2) + eps) * gain (the paper's N_e, N_h, N_o
    and the decoder's pre-norms; eps 1e-6)."""
    x = f64(x)
    return x / torch.sqrt((x * x).mean(-1, keepdim=True) + eps) * f64(gain)


def rope(x: torch.Tensor, pos: torch.Tensor, theta: float) -> torch.Tensor:
    """Rotary position embedding (RoFormer), rotate-half form over the whole head dim.

    x: [n, H, hd]; pos: [n] absolute positions.  Pair (i, i+hd/2) is rotated by the angle
    pos * theta^(-2i/hd) (Table "Model specification": theta = 1e6)."""
    x = f64(x)
    hd = x.shape[-1]
    half = hd // 2
    inv_freq = torch.tensor([theta ** (-(2.0 * i) / hd) for i in range(half)], dtype=F64)
    ang = f64(pos)[:, None] * inv_freq[None, :]
    c = torch.cos(ang)[:, None, :]
    s = torch.sin(ang)[:, None, :]
    x1, x2 = x[..., :half], x[..., half:]
    return torch.cat([x1 * c - x2 * s, x2 * c + x1 * s], dim=-1)


def attention(q: torch.Tensor, q_pos: Sequence[int], k: torch.Tensor, v: torch.Tensor) -> torch.Tensor:
    """Causal softmax attention of queries over a key/value sequence.

    q: [R, H, hd] at absolute positions q_pos; k, v: [n, H, hd] where key j sits at position j.
    Query r sees keys 0..q_pos[r]; scores are q.k / sqrt(hd).  Returns [R, H, hd]."""
    q, k, v = f64(q), f64(k), f64(v)
    R, H, hd = q.shape
    out = torch.zeros(R, H, hd, dtype=F64)
    scale = 1.0 / math.sqrt(hd)
    for r in range(R):
        n_vis = int(q_pos[r]) + 1
        for h in range(H):
            s = (k[:n_vis, h, :] @ q[r, h, :]) * scale
            p = torch.exp(s - s.max())
            p = p / p.sum()
            out[r, h] = p @ v[:n_vis, h, :]
    return out


def silu(x: torch.Tensor) -> torch.Tensor:
    return x / (1.0 + torch.exp(-x))


def swiglu(x: torch.Tensor, w_gate_up: torch.Tensor, w_down: torch.Tensor, rb: bool, fp8: bool = False) -> torch.Tensor:
    """SwiGLU FFN: W_down (silu(W_gate x) * W_up x).  w_gate_up: [2I][d], gate rows first.

    fp8=True is the fp8-expert variant (not in the paper): the weights given are the dequantised
    e4m3 matrices, and the two tensors that enter the expert products -- the input rows and the
    SwiGLU activations -- are rounded to e4m3 (instead of the activations to bf16)."""
    I = w_gate_up.shape[0] // 2
    wgu = f64(w_gate_up)
    xi = round_e4m3(f64(x)) if fp8 else f64(x)
    g = xi @ wgu[:I].T
    u = xi @ wgu[I:].T
    act = round_e4m3(silu(g) * u) if fp8 else _rb(silu(g) * u, rb)
    return act @ f64(w_down).T


def router_topk(x: torch.Tensor, w_router: torch.Tensor, top_k: int,
                bias: Optional[torch.Tensor] = None):
    """DeepSeekMoE router: p_{i,t} = softmax_i(x_t . w_i (+ bias_i)); the top_k experts by
    probability, ties to the lower expert id; gates are the selected p (no renormalisation).

    Returns (idx [n, k] int64, gates [n, k], probs [n, E], gap [n]) where gap is the
    probability margin between the k-th and (k+1)-th expert (inf when k == E)."""
    logits = f64(x) @ f64(w_router).T
    if bias is not None:
        logits = logits + f64(bias)[None, :]
    p = torch.softmax(logits, dim=-1)
    order = torch.sort(-p, dim=-1, stable=True).indices      # descending p, lower id first
    idx = order[:, :top_k]
    gates = torch.gather(p, 1, idx)
    sp = torch.gather(p, 1, order)
    if top_k < p.shape[1]:
        gap = sp[:, top_k - 1] - sp[:, top_k]
    else:
        gap = torch.full((p.shape[0],), math.inf, dtype=F64)
    return idx, gates, p, gap


def argmax_with_gap(logits: torch.Tensor):
    """Greedy token per row (lowest id among equal maxima) and the top-1 minus top-2 margin."""
    v = torch.argmax(logits, dim=-1)                 # first maximal index
    top2 = torch.topk(logits, 2, dim=-1).values
    return v, top2[:, 0] - top2[:, 1]


def accept_length(drafts: Sequence[int], v: Sequence[int]) -> int:
    """Longest equality prefix of the acceptance equation (Sec. 3.1):
    m = max({0} U {r <= K : x^_s = v_s for all s <= r}), with drafts = x^_1..x^_K and
    v = v_1..v_{K+1} (v[s-1] is the verifier token for continuation position s)."""
    m = 0
    for s in range(1, len(drafts) + 1):
        if int(drafts[s - 1]) == int(v[s - 1]):
            m = s
        else:
            break
    return m


# ----------------------------------------------------------------------------- state

@dataclass
class SeqCache:
    """Committed verifier state of one sequence: per-layer K/V for positions 0..ctx-1, and the
    pending token x_ctx (committed, not yet consumed by the verifier)."""
    k: List[torch.Tensor]          # per layer fp64 [ctx][H][hd]
    v: List[torch.Tensor]
    pending: int

    @property
    def ctx(self) -> int:
        return int(self.k[0].shape[0])

    @staticmethod
    def from_prefix(kv: torch.Tensor, pending: int) -> "SeqCache":
        """kv: bf16 [L][2][ctx][H][hd] (synthetic committed prefix, keys already rotated)."""
        return SeqCache([f64(kv[l, 0]) for l in range(kv.shape[0])],
                        [f64(kv[l, 1]) for l in range(kv.shape[0])], int(pending))


@dataclass
class DraftCache:
    """Committed draft-block KV rows 0..ctx-1 of one sequence, plus the rows that the next
    draft step must still append: the base states b_p of the newly committed rows and the
    tokens x_{p+1} that follow them (Sec. 3.1: committed rows keep their base states)."""
    k: torch.Tensor                # fp64 [ctx][H][hd]
    v: torch.Tensor
    rows_b: Optional[torch.Tensor] = None      # [n][d] base states b_p, p = ctx..ctx+n-1
    rows_tok: Optional[List[int]] = None       # [n] x_{p+1}

    @property
    def ctx(self) -> int:
        return int(self.k.shape[0])

    @staticmethod
    def from_prefix(kv: torch.Tensor) -> "DraftCache":
        return DraftCache(f64(kv[0]), f64(kv[1]))


# ----------------------------------------------------------------------------- verifier

class Verifier:
    """The MoE decoder with bf16-stored weights (synth_inputs.VerifierWeights)."""

    def __init__(self, w, shape=None):
        self.w = w
        self.s = shape if shape is not None else w.shape
        self._lm = None

    def lm_head64(self) -> torch.Tensor:
        if self._lm is None:
            self._lm = f64(self.w.lm_head)
        return self._lm

    def embed(self, tokens) -> torch.Tensor:
        return f64(self.w.embed[torch.as_tensor(list(tokens), dtype=torch.long)])


@dataclass
class VerifyOut:
    v: torch.Tensor                # int64 [B][K+1] verifier tokens v_1..v_{K+1}
    v_gap: torch.Tensor            # fp64 [B][K+1] top-1 minus top-2 logit
    m: List[int]                   # accepted draft length per sequence
    b: torch.Tensor                # [B][K+1][d] post-norm states b = N_o(h_L)
    new_k: List[List[torch.Tensor]]  # [B][L] -> [K+1][H][hd]
    new_v: List[List[torch.Tensor]]
    route_idx: List[torch.Tensor]  # per layer int64 [B*(K+1)][top_k] (row = b*(K+1)+r)
    route_gate: List[torch.Tensor]
    route_gap: List[torch.Tensor]  # per layer fp64 [B*(K+1)]
    hidden: List[torch.Tensor] = field(default_factory=list)  # per layer output h [T][d]


def _moe(model: Verifier, lw, x: torch.Tensor, rb: bool):
    """DeepSeekMoE FFN on normalised rows x [n][d]: sum over the top-k slots of gate * routed
    SwiGLU expert, plus the shared experts with gate 1, summed slot by slot."""
    s = model.s
    idx, gates, _, gap = router_topk(x, lw.router, s.top_k, lw.router_bias)
    n = x.shape[0]
    fp8 = getattr(lw, "w_gate_up_f8", None) is not None     # the fp8-expert variant
    if fp8:
        wgu = lambda e: dequant_rows(lw.w_gate_up_f8[e], lw.gate_up_scale[e])
        wdn = lambda e: dequant_rows(lw.w_down_f8[e], lw.down_scale[e])
        sgu = lambda j: dequant_rows(lw.shared_gate_up_f8[j], lw.shared_gate_up_scale[j])
        sdn = lambda j: dequant_rows(lw.shared_down_f8[j], lw.shared_down_scale[j])
    else:
        wgu, wdn = (lambda e: lw.w_gate_up[e]), (lambda e: lw.w_down[e])
        sgu, sdn = (lambda j: lw.shared_gate_up[j]), (lambda j: lw.shared_down[j])
    y_slot = torch.zeros(n, s.top_k, s.hidden, dtype=F64)
    for e in sorted(set(idx.flatten().tolist())):
        rows, slots = torch.nonzero(idx == e, as_tuple=True)
        y_slot[rows, slots] = swiglu(x[rows], wgu(e), wdn(e), rb, fp8)
    out = torch.zeros(n, s.hidden, dtype=F64)
    for k in range(s.top_k):
        out = out + gates[:, k:k + 1] * y_slot[:, k]
    for j in range(s.n_shared):
        out = out + swiglu(x, sgu(j), sdn(j), rb, fp8)
    return out, idx, gates, gap


def _attn_block(s, h, norm_w, wqkv, wo, seq_rows, keys, vals, pos, rb):
    """Pre-norm attention sublayer over several sequences.

    h [n][d] rows grouped per sequence (seq_rows[i] = list of row ids of sequence i, in
    position order), keys/vals[i] the committed K/V of sequence i, pos[i] the positions of its
    rows.  Returns (h + W_o attn, per-sequence new K, new V)."""
    H, hd = s.n_heads, s.head_dim
    x = _rb(rms_norm(h, norm_w, s.rms_eps), rb)
    qkv = x @ f64(wqkv).T
    q = qkv[:, :H * hd].reshape(-1, H, hd)
    k = qkv[:, H * hd:2 * H * hd].reshape(-1, H, hd)
    v = qkv[:, 2 * H * hd:].reshape(-1, H, hd)
    a = torch.zeros(h.shape[0], H, hd, dtype=F64)
    new_k, new_v = [], []
    for i, rows in enumerate(seq_rows):
        p = torch.as_tensor(pos[i], dtype=F64)
        qi = _rb(rope(q[rows], p, s.rope_theta), rb)
        ki = _rb(rope(k[rows], p, s.rope_theta), rb)
        vi = _rb(v[rows], rb)
        K_all = torch.cat([keys[i], ki], 0)
        V_all = torch.cat([vals[i], vi], 0)
        assert K_all.shape[0] == int(pos[i][-1]) + 1, "keys must cover positions 0..last row"
        a[rows] = attention(qi, pos[i], K_all, V_all)
        new_k.append(ki)
        new_v.append(vi)
    a = _rb(a.reshape(h.shape[0], H * hd), rb)
    return h + a @ f64(wo).T, new_k, new_v


def verify(model: Verifier, caches: Sequence[SeqCache], cand, rb: bool = True,
           keep_hidden: bool = False) -> VerifyOut:
    """Verifier forward over the K+1 candidates of every sequence, then greedy acceptance.

    cand: [B][K+1] with cand[b][0] the pending token x_c of sequence b and cand[b][1..K] its
    drafts x^_1..x^_K; candidate r sits at position c_b + r.  The state is not modified."""
    s = model.s
    cand = torch.as_tensor(cand, dtype=torch.long)
    B, R = cand.shape
    for b in range(B):
        assert int(cand[b, 0]) == caches[b].pending, "candidate 0 must be the pending token"
    h = model.embed(cand.flatten().tolist())
    seq_rows = [list(range(b * R, (b + 1) * R)) for b in range(B)]
    pos = [list(range(caches[b].ctx, caches[b].ctx + R)) for b in range(B)]
    new_k = [[None] * s.n_layers for _ in range(B)]
    new_v = [[None] * s.n_layers for _ in range(B)]
    ridx, rgate, rgap, hid = [], [], [], []
    for l, lw in enumerate(model.w.layers[:s.n_layers]):
        h, nk, nv = _attn_block(s, h, lw.attn_norm, lw.wqkv, lw.wo, seq_rows,
                                [c.k[l] for c in caches], [c.v[l] for c in caches], pos, rb)
        for b in range(B):
            new_k[b][l], new_v[b][l] = nk[b], nv[b]
        x = _rb(rms_norm(h, lw.moe_norm, s.rms_eps), rb)
        y, idx, gates, gap = _moe(model, lw, x, rb)
        h = h + y
        ridx.append(idx); rgate.append(gates); rgap.append(gap)
        if keep_hidden:
            hid.append(h.clone())
    bst = _rb(rms_norm(h, model.w.final_norm, s.rms_eps), rb)          # b = N_o(h_L)
    logits = bst @ model.lm_head64().T
    v, vgap = argmax_with_gap(logits)
    v = v.reshape(B, R)
    vgap = vgap.reshape(B, R)
    m = [accept_length(cand[b, 1:].tolist(), v[b].tolist()) for b in range(B)]
    return VerifyOut(v, vgap, m, bst.reshape(B, R, s.hidden), new_k, new_v, ridx, rgate, rgap, hid)


def commit(caches: Sequence[SeqCache], out: VerifyOut, cand, dcaches: Optional[Sequence[DraftCache]] = None):
    """Commit x^_{1:m} then v_{m+1} (Sec. 3.1): append the K/V of candidates 0..m to each
    verifier cache, drop the rejected tail, make v_{m+1} the new pending token.  When draft
    caches are given, queue the m+1 newly committed rows (base states b_p, next tokens x_{p+1})
    for the next draft step.  Returns the committed tokens per sequence."""
    cand = torch.as_tensor(cand, dtype=torch.long)
    committed = []
    for b, c in enumerate(caches):
        m = out.m[b]
        toks = [int(t) for t in cand[b, 1:m + 1].tolist()] + [int(out.v[b, m])]
        for l in range(len(c.k)):
            c.k[l] = torch.cat([c.k[l], out.new_k[b][l][:m + 1]], 0)
            c.v[l] = torch.cat([c.v[l], out.new_v[b][l][:m + 1]], 0)
        c.pending = toks[-1]
        if dcaches is not None:
            dc = dcaches[b]
            dc.rows_b = out.b[b, :m + 1].clone()
            dc.rows_tok = toks
        committed.append(toks)
    return committed


# ----------------------------------------------------------------------------- draft head

class Drafter:
    """FastMTP head: N_e, N_h, P and the shared block B_theta (synth_inputs.DraftWeights), with
    the embedding E, output norm N_o and LM head W_lm tied to the verifier's."""

    def __init__(self, dw, verifier: Verifier):
        self.dw = dw
        self.ver = verifier
        self.s = verifier.s


@dataclass
class DraftOut:
    tokens: List[List[int]]        # [B][K] drafts x^_1..x^_K of the next step
    gaps: List[List[float]]        # argmax margins per depth
    u: List[List[torch.Tensor]]    # [B][K] draft states u^(k)
    row_k: List[torch.Tensor]      # [B] committed draft K rows appended this step
    row_v: List[torch.Tensor]


def _draft_input(dr: Drafter, tok: Sequence[int], a: torch.Tensor, rb: bool) -> torch.Tensor:
    """z = P([N_e(e_{p+1}); N_h(a)]) for rows with next tokens `tok` and states a [n][d]."""
    s, dw = dr.s, dr.dw
    e = dr.ver.embed(tok)
    cat = torch.cat([_rb(rms_norm(e, dw.enorm, s.rms_eps), rb),
                     _rb(rms_norm(a, dw.hnorm, s.rms_eps), rb)], dim=-1)
    return cat @ f64(dw.eh_proj).T


def _draft_block(dr: Drafter, z: torch.Tensor, p: int, keys, vals, rb: bool):
    """u = N_o(B_theta(z; pos=p)) for one row that attends to draft rows 0..p, where keys/vals
    hold rows 0..p-1.  Returns (u, k_row, v_row)."""
    s, dw = dr.s, dr.dw
    h, nk, nv = _attn_block(s, z[None, :], dw.attn_norm, dw.wqkv, dw.wo, [[0]], [keys], [vals], [[p]], rb)
    x = _rb(rms_norm(h, dw.ffn_norm, s.rms_eps), rb)
    h = h + swiglu(x, dw.w_gate_up, dw.w_down, rb)
    u = _rb(rms_norm(h, dr.ver.w.final_norm, s.rms_eps), rb)
    return u[0], nk[0], nv[0]


def _draft_kv_rows(dr: Drafter, z: torch.Tensor, pos: Sequence[int], rb: bool):
    """B_theta's K/V for rows z [n][d] at positions pos (RoPE applied to K); the block is a
    single layer, so a row's K/V depend on its own input only."""
    s, dw = dr.s, dr.dw
    H, hd = s.n_heads, s.head_dim
    x = _rb(rms_norm(z, dw.attn_norm, s.rms_eps), rb)
    qkv = x @ f64(dw.wqkv).T
    k = qkv[:, H * hd:2 * H * hd].reshape(-1, H, hd)
    v = qkv[:, 2 * H * hd:].reshape(-1, H, hd)
    return _rb(rope(k, torch.as_tensor(list(pos), dtype=F64), s.rope_theta), rb), _rb(v, rb)


def draft(dr: Drafter, dcaches: Sequence[DraftCache], K: int, rb: bool = True) -> DraftOut:
    """One FastMTP draft step for every sequence (Sec. 3.1, Fig. "FastMTP state-shift alignment").

    The rows queued by the last commit, p = c..c+m (base states b_p, next tokens x_{p+1}),
    enter the draft cache at depth 1 (a = b_p): their K/V are committed.  The chain starts at
    the last of them, j = c+m: depth 1 at row j predicts x^_1 = x_{j+2}; depth k at row
    p = j+k-1 uses a = u^(k-1) and e = E(x^_{k-1}) and predicts x^_k = x_{j+k+1}.  Rows j+1..
    j+K-1 are tentative: they are attended to by deeper depths of this chain and then dropped."""
    s = dr.s
    W = dr.ver.lm_head64()
    toks_all, gaps_all, u_all, rk_all, rv_all = [], [], [], [], []
    for dc in dcaches:
        assert dc.rows_b is not None and len(dc.rows_tok) == dc.rows_b.shape[0] >= 1
        n = dc.rows_b.shape[0]
        c = dc.ctx
        z = _draft_input(dr, dc.rows_tok, f64(dc.rows_b), rb)
        pos = list(range(c, c + n))
        rk, rv = _draft_kv_rows(dr, z, pos, rb)
        dc.k = torch.cat([dc.k, rk], 0)                 # committed rows keep base states
        dc.v = torch.cat([dc.v, rv], 0)
        j = c + n - 1
        # depth 1 at row j: attends to committed rows 0..j (row j's own K/V is rebuilt inside)
        u, _, _ = _draft_block(dr, z[-1], j, dc.k[:j], dc.v[:j], rb)
        keys, vals = dc.k, dc.v                         # rows 0..j
        toks, gaps, us = [], [], []
        for k in range(1, K + 1):
            t, g = argmax_with_gap((u[None, :] @ W.T))
            toks.append(int(t[0])); gaps.append(float(g[0])); us.append(u)
            if k == K:
                break
            p = j + k                                   # row of depth k+1; keys hold rows 0..p-1
            z = _draft_input(dr, [toks[-1]], u[None, :], rb)[0]
            u, kr, vr = _draft_block(dr, z, p, keys, vals, rb)
            keys = torch.cat([keys, kr], 0)             # tentative row p, seen by deeper depths
            vals = torch.cat([vals, vr], 0)
        dc.rows_b, dc.rows_tok = None, None
        toks_all.append(toks); gaps_all.append(gaps); u_all.append(us)
        rk_all.append(rk); rv_all.append(rv)
    return DraftOut(toks_all, gaps_all, u_all, rk_all, rv_all)


# ----------------------------------------------------------------------------- decode loops

@dataclass
class DecodeStats:
    steps: int = 0
    committed: int = 0
    accept_hist: List[int] = field(default_factory=list)   # count of m = 0..K


def greedy_decode(model: Verifier, caches: Sequence[SeqCache], n_tokens: int, rb: bool = True):
    """Plain greedy autoregressive decoding: verify with K=0, commit v_1, repeat.
    Returns per sequence the n_tokens tokens committed after the initial pending token."""
    out = [[] for _ in caches]
    while min(len(o) for o in out) < n_tokens:
        cand = [[c.pending] for c in caches]
        vo = verify(model, caches, cand, rb)
        for b, toks in enumerate(commit(caches, vo, cand)):
            out[b].extend(toks)
    return [o[:n_tokens] for o in out]


def speculative_decode(model: Verifier, caches: Sequence[SeqCache], n_tokens: int, K: int,
                       drafter: Optional[Drafter] = None, dcaches: Optional[Sequence[DraftCache]] = None,
                       draft_fn: Optional[Callable] = None, rb: bool = True,
                       stats: Optional[DecodeStats] = None):
    """Speculative greedy decoding (Sec. 3.1).  Drafts come from the FastMTP head (drafter +
    dcaches) or from draft_fn(step, committed_so_far) -> [B][K], where committed_so_far[b] lists
    the tokens committed so far (its last entry is the pending token); losslessness holds for
    every draft.  The first step is a K=0 verify that produces the base state b the draft
    head starts from.  Returns per sequence the first n_tokens committed tokens."""
    B = len(caches)
    out = [[] for _ in range(B)]
    step = 0
    cand = [[c.pending] for c in caches]
    vo = verify(model, caches, cand, rb)
    for b, toks in enumerate(commit(caches, vo, cand, dcaches)):
        out[b].extend(toks)
    while min(len(o) for o in out) < n_tokens:
        if draft_fn is not None:
            drafts = draft_fn(step, [list(o) for o in out])
            if dcaches is not None:
                for dc in dcaches:
                    dc.rows_b, dc.rows_tok = None, None
        else:
            drafts = draft(drafter, dcaches, K, rb).tokens
        cand = [[c.pending] + list(drafts[b]) for b, c in enumerate(caches)]
        vo = verify(model, caches, cand, rb)
        for b, toks in enumerate(commit(caches, vo, cand, dcaches)):
            out[b].extend(toks)
        if stats is not None:
            stats.steps += 1
            stats.committed += sum(m + 1 for m in vo.m)
            while len(stats.accept_hist) < K + 1:
                stats.accept_hist.append(0)
            for m in vo.m:
                stats.accept_hist[m] += 1
        step += 1
    return [o[:n_tokens] for o in out]
