"""Python binding of libfastmtp.so, the C ABI in include/fastmtp.h.

Argument marshalling only: every step of the decode path runs in the library's CUDA kernels.
PyTorch provides device memory (weights, KV pools, inputs and outputs) and the stream.  There
is no fallback: if the library cannot be built or loaded, or no GPU is present, the calls
raise."""
from __future__ import annotations

import ctypes
from typing import List, Optional, Sequence

import torch

from . import build as _build

SPEC_OK, SPEC_EINVAL, SPEC_ENOMEM, SPEC_ECUDA, SPEC_ESTATE, SPEC_EDEVICE = range(6)
STATUS = {0: "SPEC_OK", 1: "SPEC_EINVAL", 2: "SPEC_ENOMEM", 3: "SPEC_ECUDA", 4: "SPEC_ESTATE", 5: "SPEC_EDEVICE"}
WS_B, WS_ROUTE_IDX, WS_ROUTE_GATE, WS_EXPERT_CNT, WS_DRAFT_U, WS_HIDDEN = range(6)

# Public entry points, in the order include/fastmtp.h declares them.
ENTRY_POINTS = ["spec_init", "spec_seq_reset", "spec_seq_set_draft_rows", "draft_step", "verify_step",
                "accept_commit", "spec_sync", "spec_seq_state", "spec_read_workspace", "spec_gemm_bf16",
                "spec_gemm_e4m3", "spec_profile", "spec_profile_read", "spec_trace_read", "spec_gemm_bf16_noalloc",
                "spec_draft_loss_workspace", "spec_draft_loss", "spec_destroy", "spec_last_error"]
KERNEL_CLASSES = ["embed", "qkv", "attention", "oproj", "router", "permute", "expert_gate_up", "expert_down",
                  "combine", "lm_head", "argmax", "commit", "draft_gemm", "draft_misc"]


class SpecConfig(ctypes.Structure):
    _fields_ = [(n, ctypes.c_int32) for n in (
        "hidden", "n_heads", "head_dim", "n_layers", "n_experts", "top_k", "n_shared", "expert_inter",
        "draft_inter", "vocab", "page_size", "max_batch", "max_pages_per_seq", "n_pages_total", "K_max",
        "max_position")] + [("rms_eps", ctypes.c_float), ("rope_theta", ctypes.c_float),
                             ("expert_fp8", ctypes.c_int32)]


class SpecLayerWeights(ctypes.Structure):
    _fields_ = [(n, ctypes.c_void_p) for n in (
        "attn_norm", "wqkv", "wo", "moe_norm", "router", "w_gate_up", "w_down", "shared_gate_up",
        "shared_down", "router_bias", "gate_up_scale", "down_scale", "shared_gate_up_scale", "shared_down_scale")]


class SpecWeights(ctypes.Structure):
    _fields_ = [("embed", ctypes.c_void_p), ("lm_head", ctypes.c_void_p), ("final_norm", ctypes.c_void_p),
                ("layers", ctypes.POINTER(SpecLayerWeights))] + [(n, ctypes.c_void_p) for n in (
                    "enorm", "hnorm", "eh_proj", "mtp_attn_norm", "mtp_wqkv", "mtp_wo", "mtp_ffn_norm",
                    "mtp_w_gate_up", "mtp_w_down")]


class SpecProfile(ctypes.Structure):
    _fields_ = [("launches", ctypes.c_int64 * len(KERNEL_CLASSES)), ("ms", ctypes.c_double * len(KERNEL_CLASSES)),
                ("experts_touched", ctypes.c_int64), ("expert_rows", ctypes.c_int64)]


class FastMTPError(RuntimeError):
    def __init__(self, status: int, msg: str):
        super().__init__(f"{STATUS.get(status, status)}: {msg}")
        self.status = status


_LIB: Optional[ctypes.CDLL] = None


def load_library(build_if_needed: bool = True) -> ctypes.CDLL:
    """Loads libfastmtp.so (building it with nvcc first when needed)."""
    global _LIB
    if _LIB is not None:
        return _LIB
    path = _build.build() if build_if_needed else _build.LIB
    lib = ctypes.CDLL(path)
    P, I32 = ctypes.c_void_p, ctypes.c_int32
    sig = {
        "spec_init": (ctypes.c_int, [ctypes.POINTER(SpecConfig), ctypes.POINTER(SpecWeights), P, P, P,
                                     ctypes.POINTER(P)]),
        "spec_seq_reset": (ctypes.c_int, [P, I32, I32, ctypes.POINTER(I32), I32]),
        "spec_seq_set_draft_rows": (ctypes.c_int, [P, I32, I32, P, ctypes.POINTER(I32)]),
        "draft_step": (ctypes.c_int, [P, I32, I32, P, P]),
        "verify_step": (ctypes.c_int, [P, I32, I32, P, P, P, P]),
        "accept_commit": (ctypes.c_int, [P, I32, P, P, P]),
        "spec_sync": (ctypes.c_int, [P]),
        "spec_seq_state": (ctypes.c_int, [P, I32, ctypes.POINTER(I32), ctypes.POINTER(I32)]),
        "spec_read_workspace": (ctypes.c_int, [P, I32, P, ctypes.c_size_t]),
        "spec_gemm_bf16": (ctypes.c_int, [P, P, P, I32, I32, I32, P]),
        "spec_gemm_e4m3": (ctypes.c_int, [P, P, P, P, I32, I32, I32, P]),
        "spec_profile": (ctypes.c_int, [P, I32]),
        "spec_profile_read": (ctypes.c_int, [P, ctypes.POINTER(SpecProfile)]),
        "spec_trace_read": (ctypes.c_int, [P, I32, I32, ctypes.POINTER(I32)]),
        "spec_gemm_bf16_noalloc": (ctypes.c_int, [P, P, P, I32, I32, I32, P]),
        "spec_draft_loss_workspace": (ctypes.c_int, [I32, I32, I32, ctypes.POINTER(ctypes.c_size_t)]),
        "spec_draft_loss": (ctypes.c_int, [P, P, P, P, P, I32, I32, I32, ctypes.c_float, ctypes.c_float,
                                           ctypes.c_float, ctypes.c_float, P, P, P, ctypes.c_size_t, P]),
        "spec_destroy": (None, [P]),
        "spec_last_error": (ctypes.c_char_p, [P]),
    }
    for name, (res, args) in sig.items():
        f = getattr(lib, name)
        f.restype = res
        f.argtypes = args
    _LIB = lib
    return lib


def _ptr(t: Optional[torch.Tensor]) -> Optional[int]:
    return None if t is None else t.data_ptr()


def _stream_handle(stream: Optional[torch.cuda.Stream]) -> int:
    s = stream if stream is not None else torch.cuda.current_stream()
    return s.cuda_stream


def gemm_bf16(X: torch.Tensor, W: torch.Tensor, stream: Optional[torch.cuda.Stream] = None) -> torch.Tensor:
    """Y = X W^T through spec_gemm_bf16 (X [M][K], W [N][K] bf16 CUDA tensors) -> fp32 [M][N]."""
    lib = load_library()
    assert X.is_cuda and W.is_cuda and X.dtype == torch.bfloat16 and W.dtype == torch.bfloat16
    X, W = X.contiguous(), W.contiguous()
    M, K = X.shape
    N = W.shape[0]
    Y = torch.empty(M, N, dtype=torch.float32, device=X.device)
    st = lib.spec_gemm_bf16(X.data_ptr(), W.data_ptr(), Y.data_ptr(), M, N, K, _stream_handle(stream))
    if st != SPEC_OK:
        raise FastMTPError(st, lib.spec_last_error(None).decode())
    return Y


def trace_read(reset: bool = True, cap: int = 3 << 16):
    """The device-timeline records of a FASTMTP_TRACE=1 build (spec_trace_read) as a uint64
    numpy array [n][4]: signature, block, t_a, t_b (see include/fastmtp.h)."""
    import numpy as np

    lib = load_library()
    buf = np.zeros((cap, 4), dtype=np.uint64)
    n = ctypes.c_int32(0)
    st = lib.spec_trace_read(buf.ctypes.data, cap, 1 if reset else 0, ctypes.byref(n))
    if st != SPEC_OK:
        raise FastMTPError(st, lib.spec_last_error(None).decode())
    return buf[: n.value].copy()


def gemm_e4m3(X8: torch.Tensor, W8: torch.Tensor, w_scale: torch.Tensor,
              stream: Optional[torch.cuda.Stream] = None) -> torch.Tensor:
    """Y = (X W^T) * w_scale through spec_gemm_e4m3 (X8 [M][K], W8 [N][K] uint8 e4m3 codes,
    w_scale fp32 [N], CUDA tensors) -> fp32 [M][N]."""
    lib = load_library()
    M, K = X8.shape
    N = W8.shape[0]
    Y = torch.empty(M, N, dtype=torch.float32, device=X8.device)
    st = lib.spec_gemm_e4m3(X8.data_ptr(), W8.data_ptr(), w_scale.data_ptr(), Y.data_ptr(), M, N, K,
                            _stream_handle(stream))
    if st != SPEC_OK:
        raise FastMTPError(st, lib.spec_last_error(None).decode())
    return Y


def gemm_bf16_noalloc(X: torch.Tensor, W: torch.Tensor, Y: torch.Tensor,
                      stream: Optional[torch.cuda.Stream] = None) -> torch.Tensor:
    """Y = X W^T through spec_gemm_bf16_noalloc (split-K with the library's fixed scratch);
    Y is a caller-provided fp32 CUDA tensor [M][N]."""
    lib = load_library()
    M, K = X.shape
    N = W.shape[0]
    assert Y.shape == (M, N) and Y.dtype == torch.float32 and Y.is_contiguous()
    st = lib.spec_gemm_bf16_noalloc(X.data_ptr(), W.data_ptr(), Y.data_ptr(), M, N, K, _stream_handle(stream))
    if st != SPEC_OK:
        raise FastMTPError(st, lib.spec_last_error(None).decode())
    return Y


def draft_loss_workspace_bytes(K: int, n_rows: int, vocab: int) -> int:
    lib = load_library()
    n = ctypes.c_size_t()
    st = lib.spec_draft_loss_workspace(K, n_rows, vocab, ctypes.byref(n))
    if st != SPEC_OK:
        raise FastMTPError(st, lib.spec_last_error(None).decode())
    return int(n.value)


def draft_loss(u: torch.Tensor, b_next: torch.Tensor, target: torch.Tensor, lm_head: torch.Tensor,
               valid: Optional[torch.Tensor] = None, beta: float = 0.6, weights=(0.85, 0.45, 0.45),
               workspace: Optional[torch.Tensor] = None, stream: Optional[torch.cuda.Stream] = None):
    """spec_draft_loss: the draft-head objective of K depths over n_rows rows.  u bf16 [K][R][d],
    b_next bf16 [R][d], target int32 [R], lm_head bf16 [V][d], valid int32 [R] or None (CUDA
    tensors).  Returns (out fp32 [1 + 3K] = L, CE_k, KL_k, MSE_k; rows fp32 [K][R][3])."""
    lib = load_library()
    K, R, d = u.shape
    V = lm_head.shape[0]
    need = draft_loss_workspace_bytes(K, R, V)
    if workspace is None:
        workspace = torch.empty(need, dtype=torch.uint8, device=u.device)
    out = torch.empty(1 + 3 * K, dtype=torch.float32, device=u.device)
    rows = torch.empty(K, R, 3, dtype=torch.float32, device=u.device)
    for t in (u, b_next, lm_head):
        assert t.dtype == torch.bfloat16 and t.is_contiguous() and t.is_cuda
    assert target.dtype == torch.int32 and target.is_contiguous()
    vp = None
    if valid is not None:
        assert valid.dtype == torch.int32 and valid.is_contiguous()
        vp = valid.data_ptr()
    st = lib.spec_draft_loss(u.data_ptr(), b_next.data_ptr(), target.data_ptr(), vp, lm_head.data_ptr(), K, R, V,
                             float(beta), float(weights[0]), float(weights[1]), float(weights[2]), out.data_ptr(),
                             rows.data_ptr(), workspace.data_ptr(), workspace.numel(), _stream_handle(stream))
    if st != SPEC_OK:
        raise FastMTPError(st, lib.spec_last_error(None).decode())
    return out, rows


def choose_depth(batch: int, ctx: int, table: Optional[dict] = None) -> int:
    """Draft depth K for a step of `batch` sequences at committed context `ctx`: the depth with
    the highest measured committed tokens/s at the nearest measured (batch, context) point of
    the draft-depth table (the packaged GB300 table unless `table` is given); 0 means plain
    greedy decoding.  Host-side only: no library call."""
    from . import depth_table as _dt
    from . import metrics as _m
    pol = _m.DepthPolicy.from_table(table if table is not None else _dt.load_packaged())
    return pol.choose(int(batch), int(ctx))


def device_sync() -> None:
    """spec_sync(NULL): waits for the current device and raises FastMTPError (SPEC_EDEVICE) if a
    kernel of spec_gemm_bf16 or spec_gemm_bf16_noalloc set its guard flag since the last check."""
    lib = load_library()
    st = lib.spec_sync(None)
    if st != SPEC_OK:
        raise FastMTPError(st, lib.spec_last_error(None).decode())


class Engine:
    """A spec_ctx with device copies of the verifier and draft weights and the two KV pools.

    vw / dw: synth_inputs.VerifierWeights / DraftWeights (bf16 CPU tensors).  Slot b owns pages
    b*max_pages_per_seq .. (b+1)*max_pages_per_seq-1 of both pools."""

    def __init__(self, vw, dw, max_batch: int, K_max: int, max_ctx: int, page_size: int = 64,
                 device: str = "cuda", stream: Optional[torch.cuda.Stream] = None, max_position: int = 32768,
                 expert_fp8: bool = False):
        self.lib = load_library()
        if not torch.cuda.is_available():
            raise RuntimeError("FastMTP needs a CUDA GPU")
        s = vw.shape
        self.shape = s
        self.device = torch.device(device)
        self.stream = stream if stream is not None else torch.cuda.current_stream(self.device)
        self.page_size = page_size
        self.max_batch = max_batch
        self.K_max = K_max
        self.max_pages = (max_ctx + K_max + 1 + page_size - 1) // page_size
        self.n_pages = max_batch * self.max_pages
        dev = lambda t: t.to(self.device).contiguous()
        self._keep: List[torch.Tensor] = []

        def keep(t):
            t = dev(t)
            self._keep.append(t)
            return t

        self.embed = keep(vw.embed)
        self.lm_head = keep(vw.lm_head)
        final_norm = keep(vw.final_norm)
        self._layers = (SpecLayerWeights * s.n_layers)()
        for l, lw in enumerate(vw.layers[:s.n_layers]):
            L = self._layers[l]
            L.attn_norm = keep(lw.attn_norm).data_ptr()
            L.wqkv = keep(lw.wqkv).data_ptr()
            L.wo = keep(lw.wo).data_ptr()
            L.moe_norm = keep(lw.moe_norm).data_ptr()
            L.router = keep(lw.router).data_ptr()
            if expert_fp8:   # e4m3 codes with one fp32 scale per row (synth_inputs.quantize_experts_fp8)
                L.w_gate_up = keep(lw.w_gate_up_f8).data_ptr()
                L.w_down = keep(lw.w_down_f8).data_ptr()
                L.shared_gate_up = keep(lw.shared_gate_up_f8).data_ptr()
                L.shared_down = keep(lw.shared_down_f8).data_ptr()
                L.gate_up_scale = keep(lw.gate_up_scale.float()).data_ptr()
                L.down_scale = keep(lw.down_scale.float()).data_ptr()
                L.shared_gate_up_scale = keep(lw.shared_gate_up_scale.float()).data_ptr()
                L.shared_down_scale = keep(lw.shared_down_scale.float()).data_ptr()
            else:
                L.w_gate_up = keep(lw.w_gate_up).data_ptr()
                L.w_down = keep(lw.w_down).data_ptr()
                L.shared_gate_up = keep(lw.shared_gate_up).data_ptr()
                L.shared_down = keep(lw.shared_down).data_ptr()
            L.router_bias = keep(lw.router_bias.float()).data_ptr() if lw.router_bias is not None else None
        w = SpecWeights()
        w.embed, w.lm_head, w.final_norm = self.embed.data_ptr(), self.lm_head.data_ptr(), final_norm.data_ptr()
        w.layers = self._layers
        for name in ("enorm", "hnorm", "eh_proj"):
            setattr(w, name, keep(getattr(dw, name)).data_ptr())
        for name in ("attn_norm", "wqkv", "wo", "ffn_norm", "w_gate_up", "w_down"):
            setattr(w, "mtp_" + name, keep(getattr(dw, name)).data_ptr())
        self._w = w
        H, hd = s.n_heads, s.head_dim
        self.kv_pool = torch.zeros(s.n_layers, self.n_pages, 2, H, page_size, hd, dtype=torch.bfloat16,
                                   device=self.device)
        self.dkv_pool = torch.zeros(self.n_pages, 2, H, page_size, hd, dtype=torch.bfloat16, device=self.device)
        cfg = SpecConfig(hidden=s.hidden, n_heads=H, head_dim=hd, n_layers=s.n_layers, n_experts=s.n_experts,
                         top_k=s.top_k, n_shared=s.n_shared, expert_inter=s.expert_inter,
                         draft_inter=s.draft_inter, vocab=s.vocab, page_size=page_size, max_batch=max_batch,
                         max_pages_per_seq=self.max_pages, n_pages_total=self.n_pages, K_max=K_max,
                         max_position=max_position, rms_eps=s.rms_eps, rope_theta=s.rope_theta,
                         expert_fp8=1 if expert_fp8 else 0)
        self._cfg = cfg
        ctx = ctypes.c_void_p()
        torch.cuda.synchronize(self.device)
        st = self.lib.spec_init(ctypes.byref(cfg), ctypes.byref(w), self.kv_pool.data_ptr(), self.dkv_pool.data_ptr(),
                                self.stream.cuda_stream, ctypes.byref(ctx))
        if st != SPEC_OK:
            raise FastMTPError(st, self.lib.spec_last_error(None).decode())
        self.ctx = ctx

    # ------------------------------------------------------------------ helpers
    def _check(self, st: int):
        if st != SPEC_OK:
            raise FastMTPError(st, self.lib.spec_last_error(self.ctx).decode())

    def block_table(self, slot: int) -> List[int]:
        return [slot * self.max_pages + i for i in range(self.max_pages)]

    def load_prefix(self, slot: int, kv: Optional[torch.Tensor], dkv: Optional[torch.Tensor], pending: int,
                    ctx_len: Optional[int] = None):
        """Places a synthetic committed prefix in slot `slot`'s pages and resets the slot.
        kv: bf16 [L][2][ctx][H][hd] (verifier rows) or None; dkv: bf16 [2][ctx'][H][hd] (draft rows)
        or None; ctx_len defaults to the verifier prefix length."""
        ps = self.page_size
        bt = self.block_table(slot)
        if kv is not None:
            ctx = kv.shape[2]
            n = (ctx + ps - 1) // ps
            if n:
                src = torch.nn.functional.pad(kv.to(self.device), (0, 0, 0, 0, 0, n * ps - ctx))
                src = src.reshape(kv.shape[0], 2, n, ps, kv.shape[3], kv.shape[4]).permute(0, 2, 1, 4, 3, 5)
                self.kv_pool[:, bt[0]:bt[0] + n] = src
        if dkv is not None:
            ctx = dkv.shape[1]
            n = (ctx + ps - 1) // ps
            if n:
                dsrc = torch.nn.functional.pad(dkv.to(self.device), (0, 0, 0, 0, 0, n * ps - ctx))
                dsrc = dsrc.reshape(2, n, ps, dkv.shape[2], dkv.shape[3]).permute(1, 0, 3, 2, 4)
                self.dkv_pool[bt[0]:bt[0] + n] = dsrc
        if ctx_len is None:
            ctx_len = kv.shape[2] if kv is not None else dkv.shape[1]
        torch.cuda.synchronize(self.device)
        self.reset_seq(slot, ctx_len, bt, pending)

    def reset_seq(self, slot: int, ctx_len: int, block_table: Sequence[int], pending: int):
        arr = (ctypes.c_int32 * self.max_pages)(*list(block_table))
        self._check(self.lib.spec_seq_reset(self.ctx, slot, ctx_len, arr, pending))

    def set_draft_rows(self, slot: int, b_rows: torch.Tensor, next_tokens: Sequence[int]):
        b_rows = b_rows.to(self.device, torch.bfloat16).contiguous()
        arr = (ctypes.c_int32 * len(next_tokens))(*[int(t) for t in next_tokens])
        self._check(self.lib.spec_seq_set_draft_rows(self.ctx, slot, len(next_tokens), b_rows.data_ptr(), arr))

    def seq_state(self, slot: int):
        a, b = ctypes.c_int32(), ctypes.c_int32()
        self._check(self.lib.spec_seq_state(self.ctx, slot, ctypes.byref(a), ctypes.byref(b)))
        return a.value, b.value

    # ------------------------------------------------------------------ the step
    def draft_step(self, slots: torch.Tensor, K: int, cand: torch.Tensor):
        self._check(self.lib.draft_step(self.ctx, slots.numel(), K, slots.data_ptr(), cand.data_ptr()))

    def verify_step(self, slots: torch.Tensor, cand: torch.Tensor, vtok: torch.Tensor, accept: torch.Tensor):
        K = cand.shape[1] - 1
        self._check(self.lib.verify_step(self.ctx, slots.numel(), K, slots.data_ptr(), cand.data_ptr(),
                                         vtok.data_ptr(), accept.data_ptr()))

    def accept_commit(self, slots: torch.Tensor, committed: torch.Tensor, n_committed: torch.Tensor):
        self._check(self.lib.accept_commit(self.ctx, slots.numel(), slots.data_ptr(), committed.data_ptr(),
                                           n_committed.data_ptr()))

    def sync(self):
        self._check(self.lib.spec_sync(self.ctx))

    def read_workspace(self, which: int, shape, dtype) -> torch.Tensor:
        out = torch.empty(*shape, dtype=dtype)
        self._check(self.lib.spec_read_workspace(self.ctx, which, out.data_ptr(), out.numel() * out.element_size()))
        return out

    def profile(self, mode: int):
        """1: zero the counters and time every launch group; 2: zero the counters only; 0: stop."""
        self._check(self.lib.spec_profile(self.ctx, int(mode)))

    def profile_read(self) -> dict:
        p = SpecProfile()
        self._check(self.lib.spec_profile_read(self.ctx, ctypes.byref(p)))
        return {"launches": {k: int(p.launches[i]) for i, k in enumerate(KERNEL_CLASSES)},
                "ms": {k: float(p.ms[i]) for i, k in enumerate(KERNEL_CLASSES)},
                "experts_touched": int(p.experts_touched), "expert_rows": int(p.expert_rows)}

    def close(self):
        if getattr(self, "ctx", None):
            self.lib.spec_destroy(self.ctx)
            self.ctx = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass
