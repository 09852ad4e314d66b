"""Device timeline of a FASTMTP_TRACE=1 build: from the per-CTA records of spec_trace_read
(entry, wait return, exit; include/fastmtp.h) to launches and the time breakdown of one verify
layer.

Grouping: a kernel is launched only after every CTA of the previous kernel has entered (each
triggers its dependents at entry), so no other kernel's CTA enters between two CTA entries of
one launch; the records of one kernel are split into launches exactly where another kernel's
entry falls between two of theirs.  This holds for launches that run in several waves, whose
late CTAs enter long after the first ones.

A launch's `ready` time is the first wait return of its CTAs (the moment the previous kernel's
results are visible to it), its `done` time the last exit record of its CTAs.  The layer
breakdown gives, for each kernel of a verify layer, ready -> done and the hand-over from the
previous kernel's done to its ready.  Kernels without exit records (embedding, RMSNorm, commit,
draft glue) get done = the next launch's ready.
"""
from __future__ import annotations

from typing import Dict, List, Sequence

import numpy as np

EXIT_BIT = 1 << 63
KERNEL_NAMES = {1: "gemm_f32", 2: "gemm_resid", 3: "gemm_qkv", 4: "gemm_swiglu", 5: "gemm_scatter",
                6: "lm_head_argmax", 7: "experts", 16: "attention", 17: "router", 18: "combine",
                19: "embed", 20: "rmsnorm", 21: "commit", 22: "draft_prep", 23: "gather_rows",
                24: "draft_next"}
# the kernels of one verify layer, in launch order (QKV, attention, O-proj, router, experts, combine)
VERIFY_LAYER = (3, 16, 2, 17, 7, 18)


def _sig_fields(sig: int) -> Dict[str, int]:
    return {"kid": (sig >> 48) & 0x7FFF, "grid_x": (sig >> 32) & 0xFFFF, "grid_y": (sig >> 16) & 0xFFFF,
            "block": sig & 0xFFFF}


def launches(records: np.ndarray) -> List[Dict[str, object]]:
    """Groups the records into launches, in the order their inputs became ready.  Times are in
    microseconds from the first entry of the trace."""
    r = np.asarray(records, dtype=np.uint64).reshape(-1, 4)
    if len(r) == 0:
        return []
    sig = r[:, 0].astype(object)
    is_exit = np.array([int(s) & EXIT_BIT != 0 for s in sig], dtype=bool)
    base = np.array([int(s) & ~EXIT_BIT for s in sig], dtype=object)
    t0 = int(r[~is_exit, 2].min()) if (~is_exit).any() else int(r[:, 2].min())
    entries = r[~is_exit, 2].astype(np.int64)
    entry_sig = base[~is_exit]
    out = []
    for s in sorted(set(entry_sig)):
        m = (base == s) & ~is_exit
        rows = r[m]
        rows = rows[np.argsort(rows[:, 2].astype(np.int64), kind="stable")]
        ta = rows[:, 2].astype(np.int64)
        others = np.sort(entries[entry_sig != s])
        # a cut between consecutive entries of this kernel if another kernel's entry lies
        # strictly between them
        lo = np.searchsorted(others, ta[:-1], side="right")
        hi = np.searchsorted(others, ta[1:], side="left")
        cuts = [0] + [i + 1 for i in np.nonzero(hi > lo)[0].tolist()] + [len(ta)]
        ex = np.sort(r[(base == s) & is_exit][:, 2].astype(np.int64))
        groups = []
        for j in range(len(cuts) - 1):
            g = rows[cuts[j]:cuts[j + 1]]
            groups.append({"sig": int(s), **_sig_fields(int(s)), "ctas": int(len(g)),
                           "entry": (int(g[:, 2].astype(np.int64).min()) - t0, int(g[:, 2].astype(np.int64).max()) - t0),
                           "ready": (int(g[:, 3].astype(np.int64).min()) - t0, int(g[:, 3].astype(np.int64).max()) - t0),
                           "done": None})
        # exit records belong to the launch whose ready time precedes them most closely
        for k, g in enumerate(groups):
            lo = g["ready"][0] + t0
            hi = groups[k + 1]["ready"][0] + t0 if k + 1 < len(groups) else None
            e = ex[(ex >= lo) & ((ex < hi) if hi is not None else True)]
            if len(e):
                g["done"] = (int(e.min()) - t0, int(e.max()) - t0)
        out.extend(groups)
    out.sort(key=lambda g: g["ready"][0])
    for k, g in enumerate(out):
        g["name"] = KERNEL_NAMES.get(g["kid"], f"kernel{g['kid']}")
        if g["done"] is None and k + 1 < len(out):
            g["done_from_next"] = True
            g["done"] = (out[k + 1]["ready"][0], out[k + 1]["ready"][0])
        for key in ("entry", "ready", "done"):
            if g[key] is not None:
                g[key] = (g[key][0] / 1e3, g[key][1] / 1e3)
    return out


def verify_layers(ls: Sequence[Dict[str, object]]) -> List[List[Dict[str, object]]]:
    """The launches of every verify layer: consecutive runs matching VERIFY_LAYER."""
    kids = [g["kid"] for g in ls]
    n = len(VERIFY_LAYER)
    layers, i = [], 0
    while i + n <= len(ls):
        if tuple(kids[i:i + n]) == VERIFY_LAYER:
            layers.append(list(ls[i:i + n]))
            i += n
        else:
            i += 1
    return layers


def layer_breakdown(layers: Sequence[Sequence[Dict[str, object]]], skip_first: bool = True) -> Dict[str, float]:
    """Mean over verify layers (the first skipped: it follows the embedding, not a combine) of
    each kernel's ready -> done time and of the hand-over gap before it, in microseconds."""
    acc: Dict[str, List[float]] = {}
    for idx, layer in enumerate(layers):
        if skip_first and idx == 0 and len(layers) > 1:
            continue
        prev = layers[idx - 1][-1] if idx > 0 else None
        prev_done = prev["done"][1] if (prev is not None and prev["done"] is not None) else None
        for g in layer:
            if g["done"] is not None:
                acc.setdefault(g["name"], []).append(g["done"][1] - g["ready"][0])
            if prev_done is not None:
                acc.setdefault("gap_before_" + g["name"], []).append(g["ready"][0] - prev_done)
            prev_done = g["done"][1] if g["done"] is not None else None
        if layer[-1]["done"] is not None:
            acc.setdefault("layer", []).append(layer[-1]["done"][1] - layer[0]["ready"][0])
    return {k: float(np.mean(v)) for k, v in acc.items()}
