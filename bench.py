#!/usr/bin/env python
"""Benchmark of the FastMTP speculative decode step on GB300.

One step = draft_step + verify_step + accept_commit (every row of the hot path) over one
batch.  Workload: the 12-layer MoE verifier at the paper's widths (d=1280, 10x128 heads, 64
routed + 2 shared experts, top-6, vocabulary 129,280) with the FastMTP draft block
(intermediate 3584), batch 8, K = 3 drafts, committed contexts U[768, 1024] of which the first
256 positions stand in for the visual tokens.  Weights are seeded random-init bf16 ~N(0, 0.02),
KV prefixes seeded N(0, 1); nothing is read from a dataset.

Metric: accepted (committed) tokens per second, sum over sequences of (m + 1) per step,
whole job over all GPUs.  Prints one JSON line (rank 0).

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl fastmtp|reference]
  python bench.py --sweep [--sweep-batch 1,4,16,64,256] [--sweep-ctx 1024,4096,8192]
                  [--sweep-k 0,1,2,3] [--sweep-router uniform,zipf]
  python bench.py --trace [--batch B --ctx-lo C --ctx-hi C]

`--impl reference` times the fp64 CPU oracle on a bounded sample of the same workload (the
method's only other implementation here); under torchrun only rank 0 runs it.  `--sweep`
measures the step at every (batch, context, K, router) point of the verify-throughput grid,
one JSON line per point (one GPU); K = 0 is greedy decoding, the baseline of the speedup S.
`--trace` prints the device timeline of one step (every launch and the breakdown of a verify
layer) from the FASTMTP_TRACE=1 build of the library; it is not a timing run.
"""
from __future__ import annotations

import argparse
import hashlib
import json
import os
import statistics
import subprocess
import sys
import tempfile
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "accepted tokens/sec at batch 1–256 (K=3); verify-step HBM-roofline fraction"
WORKLOAD = ("12-layer MoE verifier (d=1280, 10x128 heads, 64 routed + 2 shared experts top-6, I=896, "
            "vocab 129280) + FastMTP draft block (I=3584); B=8, K=3, context U[768,1024] with a 256-token "
            "synthetic visual prefix; one step = draft_step + verify_step + accept_commit")
ACCEPT_RATIO = 7.0   # beta/alpha of the successor-map weights: tau ~2.7 (the paper's k=3 operating point)
FALLBACK_HBM_GBS = 6800.0


def parse():
    import synth_inputs as S
    c1, c4 = S.WORKLOADS["verify_12l_b8_ctx768_1024"], S.WORKLOADS["sweep_12l_b1_256_ctx1024_8192"]
    p = argparse.ArgumentParser()
    p.add_argument("--gpus", type=int, default=1)
    p.add_argument("--steps", type=int, default=20)
    p.add_argument("--warmup", type=int, default=5)
    p.add_argument("--impl", default="fastmtp", choices=["fastmtp", "reference"])
    p.add_argument("--batch", type=int, default=c1.batch)
    p.add_argument("--K", type=int, default=c1.K)
    p.add_argument("--ctx-lo", type=int, default=c1.ctx_lo)
    p.add_argument("--ctx-hi", type=int, default=c1.ctx_hi)
    p.add_argument("--layers", type=int, default=c1.n_layers)
    p.add_argument("--seed", type=int, default=c1.seed)
    p.add_argument("--cpu-budget-s", type=float, default=20.0, help="CPU seconds of the oracle sample")
    p.add_argument("--no-cpu-baseline", action="store_true")
    p.add_argument("--no-e2e", action="store_true")
    p.add_argument("--no-points", action="store_true",
                   help="skip the B=1/64/256 points of the metric's batch range (ctx 1024, K=3)")
    p.add_argument("--weights", default="successor", choices=["successor", "random"],
                   help="successor: acceptance-tuned seeded weights (tau ~2.7); random: N(0,0.02) everywhere")
    p.add_argument("--device-kv", action="store_true",
                   help="draw the KV prefixes on the GPU (PyTorch's generator) instead of the host Philox stream")
    p.add_argument("--sweep", action="store_true", help="run the (batch, context, K, router) grid")
    p.add_argument("--experts", default="bf16", choices=["bf16", "fp8"],
                   help="fp8: the fp8-expert variant (e4m3 expert matrices with per-row scales) as the main "
                        "workload; the default bf16 is the paper's model")
    p.add_argument("--objective", action="store_true",
                   help="time only the draft-head training objective (64 rows, K=3, full vocabulary)")
    p.add_argument("--trace", action="store_true",
                   help="device timeline of one step (builds the FASTMTP_TRACE=1 library): every launch "
                        "and the per-kernel breakdown of a verify layer, as JSON lines")
    p.add_argument("--trace-out", default="", help="with --trace: also save the raw records (.npy, uint64 [n][4])")
    p.add_argument("--sweep-batch", default=",".join(map(str, c4.grid["batch"])))
    p.add_argument("--sweep-ctx", default=",".join(map(str, c4.grid["ctx"])))
    p.add_argument("--sweep-k", default=",".join(map(str, c4.grid["K"])),
                   help="draft depths; 0 = greedy decoding, the speedup baseline")
    p.add_argument("--sweep-router", default=",".join(c4.grid["router"]))
    return p.parse_args()


def measured_peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        d = json.load(open(path))
        return float(d["hbm_gbs"]), "measured"
    except Exception:
        return FALLBACK_HBM_GBS, "fallback"


# ----------------------------------------------------------------------------- workload
def data_desc(args):
    if args.weights == "successor":
        return (f"synthetic: seeded acceptance-tuned weights (successor map, beta/alpha={ACCEPT_RATIO}), "
                "other matrices N(0,0.02), N(0,1) KV prefixes")
    return "synthetic: seeded random-init weights N(0,0.02), N(0,1) KV prefixes"


def rank_seed(seed, rank):
    """Replica r draws its own sequences (contexts, pending tokens, KV prefixes) from seed + 1000 r;
    the weights are the same on every replica."""
    return seed + 1000 * rank


def sequence_inputs(args, shape, rank=0):
    """Contexts and pending tokens of the replica's B sequences (host, cheap)."""
    import synth_inputs as S
    sd = rank_seed(args.seed, rank)
    ctx = [int(c) for c in S.integers(sd, "ctx", args.batch, args.ctx_lo, args.ctx_hi)]
    pend = [int(t) for t in S.integers(sd, "pending", args.batch, 0, shape.vocab - 1)]
    return ctx, pend


def workload(args, rank=0):
    import synth_inputs as S
    shape = S.ModelShape(n_layers=args.layers)
    seed = args.seed
    if args.weights == "successor":
        vw, dw, _ = S.successor_weights(shape, seed, ACCEPT_RATIO)
    else:
        vw = S.verifier_weights(shape, seed)
        dw = S.draft_weights(shape, seed)
    if getattr(args, "experts", "bf16") == "fp8":
        vw = S.quantize_experts_fp8(vw)
    B = args.batch
    ctx, pend = sequence_inputs(args, shape, rank)
    sd = rank_seed(seed, rank)
    if args.device_kv:
        dev = f"cuda:{int(os.environ.get('LOCAL_RANK', '0'))}"
        kvs = [S.kv_prefix_device(sd, b, shape.n_layers, ctx[b], shape.n_heads, shape.head_dim, dev) for b in range(B)]
        dkvs = [S.draft_kv_prefix_device(sd, b, ctx[b], shape.n_heads, shape.head_dim, dev) for b in range(B)]
    else:
        kvs = [S.kv_prefix(sd, b, shape.n_layers, ctx[b], shape.n_heads, shape.head_dim) for b in range(B)]
        dkvs = [S.draft_kv_prefix(sd, b, ctx[b], shape.n_heads, shape.head_dim) for b in range(B)]
    return shape, vw, dw, ctx, pend, kvs, dkvs


def job_totals(ms, tokens, world, device):
    """Whole-job (time, tokens) of the replicas: the slowest rank's time and the sum of the
    committed tokens (a collective over the default process group when world > 1)."""
    if world <= 1:
        return float(ms), int(tokens)
    import torch
    import torch.distributed as dist
    t = torch.tensor([float(ms)], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    n = torch.tensor([int(tokens)], dtype=torch.int64, device=device)
    dist.all_reduce(n, op=dist.ReduceOp.SUM)
    return float(t.item()), int(n.item())


def algorithmic_bytes(shape, B, K, ctx_mean, experts_touched_routed_per_layer, fp8_experts=False):
    """Bytes the verify step must move: every weight matrix it reads once (routed experts counted
    from the actual routing; e4m3 experts one byte per weight plus an fp32 scale per row), the
    committed KV it reads, the candidate KV it writes and the embedding rows."""
    d, H, hd, I, E, L, V = (shape.hidden, shape.n_heads, shape.head_dim, shape.expert_inter, shape.n_experts,
                            shape.n_layers, shape.vocab)
    T = B * (K + 1)
    attn_w = 2 * (3 * H * hd * d + d * H * hd)
    router_w = 2 * E * d
    expert_w = (3 * d * I + 4 * (2 * I + d)) if fp8_experts else 2 * 3 * d * I
    shared_w = shape.n_shared * expert_w
    kv_tok = 2 * H * hd * 2
    per_layer = attn_w + router_w + shared_w + expert_w * experts_touched_routed_per_layer
    return L * per_layer + 2 * V * d + B * ctx_mean * L * kv_tok + T * L * kv_tok + T * d * 2


def draft_algorithmic_bytes(shape, B, K, ctx_mean, rows_new):
    """Bytes one draft step must move: per depth the projection P, the block B_theta's four
    matrices and the tied LM head (each read once), and the draft cache rows every sequence's
    query attends to; plus the K/V rows the depth-1 pass commits and the embedding rows read."""
    d, H, hd, Id, V = shape.hidden, shape.n_heads, shape.head_dim, shape.draft_inter, shape.vocab
    P = 2 * d * 2 * d
    block = 2 * (3 * H * hd * d + d * H * hd + 2 * Id * d + d * Id)
    lm = 2 * V * d
    kv_row = 2 * H * hd * 2
    return K * (P + block + lm) + K * B * ctx_mean * kv_row + rows_new * kv_row + (rows_new + B * K) * d * 2


# ----------------------------------------------------------------------------- clocks
class ClockSampler:
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index):
        self.gpu = gpu_index
        self.proc = None
        self.path = None

    def start(self):
        try:
            fd, self.path = tempfile.mkstemp(suffix=".csv")
            os.close(fd)
            self.proc = subprocess.Popen(["nvidia-smi", "-i", str(self.gpu), f"--query-gpu={self.FIELDS}",
                                          "--format=csv,noheader,nounits", "-lms", "200"],
                                         stdout=open(self.path, "w"), stderr=subprocess.DEVNULL)
        except Exception:
            self.proc = None

    def stop(self):
        if self.proc is None:
            return None
        time.sleep(0.25)
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except Exception:
            self.proc.kill()
        rows = []
        for line in open(self.path):
            f = [x.strip() for x in line.split(",")]
            if len(f) < 9:
                continue
            try:
                rows.append((float(f[1]), float(f[2]), f[4], f[5], f[6], f[7], f[8]))
            except ValueError:
                continue
        os.unlink(self.path)
        if not rows:
            return None
        reasons = set()
        names = ("hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap")
        for r in rows:
            for n, v in zip(names, r[3:]):
                if v.lower() == "active":
                    reasons.add(n)
        return {"sm_mhz": statistics.median(r[0] for r in rows), "sm_max_mhz": max(r[1] for r in rows),
                "reasons": sorted(reasons), "samples": len(rows)}


# ----------------------------------------------------------------------------- oracle leg
class OracleRunner:
    """The fp64 oracle on the host cores, run on the workload's first sequence: speculative
    steps of draft (K) + verify + commit, after one untimed K=0 step that gives the first base
    state."""

    def __init__(self, args, shape, vw, dw, ctx, pend, kvs, dkvs):
        import oracle as O
        self.O = O
        self.K = args.K
        self.model = O.Verifier(vw)
        self.dr = O.Drafter(dw, self.model)
        self.cache = O.SeqCache.from_prefix(kvs[0].cpu(), pend[0])
        self.dcache = O.DraftCache.from_prefix(dkvs[0].cpu())
        vo = O.verify(self.model, [self.cache], [[self.cache.pending]], rb=True)
        O.commit([self.cache], vo, [[self.cache.pending]], [self.dcache])

    def step(self):
        O = self.O
        drafts = O.draft(self.dr, [self.dcache], self.K, rb=True).tokens[0]
        cand = [[self.cache.pending] + drafts]
        vo = O.verify(self.model, [self.cache], cand, rb=True)
        return len(O.commit([self.cache], vo, cand, [self.dcache])[0])


def cpu_oracle_sample(args, work, budget_s):
    """Oracle speculative steps until about budget_s seconds have been spent."""
    import torch
    run = OracleRunner(args, *work)
    tokens, steps = 0, 0
    t0 = time.perf_counter()
    while True:
        tokens += run.step()
        steps += 1
        if time.perf_counter() - t0 >= budget_s:
            break
    dt = time.perf_counter() - t0
    return {"value": tokens / dt, "unit": "tokens/s", "cores": torch.get_num_threads(), "kind": "oracle",
            "sample": f"{steps} speculative steps (draft K={args.K} + verify + commit) of sequence 0 of the "
                      f"B={args.batch} workload, fp64, {dt:.1f} s"}


def run_reference(args):
    import torch
    if int(os.environ.get("RANK", "0")) != 0:
        return
    work = workload(args)
    run = OracleRunner(args, *work)
    for _ in range(min(args.warmup, 1)):
        run.step()
    per, tok = [], 0
    for _ in range(args.steps):
        t0 = time.perf_counter()
        tok += run.step()
        per.append(time.perf_counter() - t0)
    value = tok / sum(per)
    cores = torch.get_num_threads()
    sample = (f"{args.steps} timed speculative steps (draft K={args.K} + verify + commit) of sequence 0 of the "
              f"B={args.batch} workload, fp64")
    out = {"metric": METRIC, "impl": "reference", "value": value, "unit": "tokens/s", "n_gpus": args.gpus,
           "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1000 * statistics.mean(per),
           "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
           "data": data_desc(args),
           "config": {"workload": WORKLOAD, "batch": args.batch, "K": args.K, "layers": args.layers,
                      "weights": args.weights, "sample": "sequence 0 of the batch"},
           "cpu_baseline": {"value": value, "unit": "tokens/s", "cores": cores, "kind": "oracle", "sample": sample},
           "e2e": {"value": value, "unit": "tokens/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(out), flush=True)


# ----------------------------------------------------------------------------- GPU leg
POINT_BATCHES = (1, 64, 256)
POINT_CTX = 1024


def run_points(args, shape, vw, dw, dev, peak, peak_kind):
    """The metric's batch range on the same weights: uniform routing, K = 3, committed contexts
    of exactly 1024 tokens (N(0,1) KV drawn on the device), B = 1, 64 and 256 on one engine.
    Per point: one K=0 step, `warmup` steps, then timed steps (50 at B = 1, whose acceptance
    varies most from step to step; `steps` otherwise) with an event pair around each phase;
    per-step medians.  Returns one object per point."""
    import torch

    from paper_2609_03181_gb300 import fastmtp as F

    K, L = 3, shape.n_layers
    n_steps = {b: (max(args.steps, 50) if b == 1 else args.steps) for b in POINT_BATCHES}
    grow = (args.warmup + max(n_steps.values()) + 2) * (K + 1)
    Bmax = max(POINT_BATCHES)
    stream = torch.cuda.Stream(dev)
    eng = F.Engine(vw, dw, max_batch=Bmax, K_max=K, max_ctx=POINT_CTX + grow, page_size=64, device=str(dev),
                   stream=stream)
    g = torch.Generator(device=dev)
    g.manual_seed(4)
    for l in range(L):
        eng.kv_pool[l].normal_(generator=g)
    eng.dkv_pool.normal_(generator=g)
    torch.cuda.synchronize(dev)
    out = []
    for bi, B in enumerate(POINT_BATCHES):
        import synth_inputs as S
        pend = [int(t) for t in S.integers(40 + bi, "pending", B, 0, shape.vocab - 1)]
        for b in range(B):
            eng.reset_seq(b, POINT_CTX, eng.block_table(b), pend[b])
        slots = torch.arange(B, dtype=torch.int32, device=dev)
        c0 = torch.tensor([[p] for p in pend], dtype=torch.int32, device=dev)
        v0 = torch.empty(B, 1, dtype=torch.int32, device=dev)
        acc = torch.empty(B, dtype=torch.int32, device=dev)
        cand = torch.empty(B, K + 1, dtype=torch.int32, device=dev)
        vt = torch.empty(B, K + 1, dtype=torch.int32, device=dev)
        com = torch.empty(B, K + 1, dtype=torch.int32, device=dev)
        n_all = args.warmup + n_steps[B]
        hist = torch.zeros(n_all, B, dtype=torch.int32, device=dev)
        ev = [[torch.cuda.Event(enable_timing=True) for _ in range(4)] for _ in range(n_all)]
        torch.cuda.synchronize(dev)
        with torch.cuda.stream(stream):
            eng.verify_step(slots, c0, v0, acc)
            eng.accept_commit(slots, v0, acc)
            for i in range(n_all):
                if i == args.warmup:
                    eng.profile(2)
                ev[i][0].record(stream)
                eng.draft_step(slots, K, cand)
                ev[i][1].record(stream)
                eng.verify_step(slots, cand, vt, acc)
                ev[i][2].record(stream)
                eng.accept_commit(slots, com, hist[i])
                ev[i][3].record(stream)
        eng.sync()
        counted = eng.profile_read()
        eng.profile(0)
        timed = range(args.warmup, n_all)
        med = lambda a, b: statistics.median(ev[i][a].elapsed_time(ev[i][b]) for i in timed)
        ms_step, ms_draft, ms_verify = med(0, 3), med(0, 1), med(1, 2)
        h = hist.double().cpu()
        lens = POINT_CTX + 1 + torch.cumsum(h, 0) - h
        ctx_mean = float(lens[args.warmup:].mean())
        tok = float(h[args.warmup:].sum())
        nt = n_steps[B]
        touched = counted["experts_touched"] / max(1, counted["launches"]["router"])
        vbytes = algorithmic_bytes(shape, B, K, ctx_mean, touched - shape.n_shared)
        dbytes = draft_algorithmic_bytes(shape, B, K, ctx_mean, tok / nt)
        out.append({"batch": B, "ctx": POINT_CTX, "K": K, "K_policy": F.choose_depth(B, POINT_CTX),
                    "router": "uniform", "steps": nt,
                    "tokens_per_s": tok / (ms_step * nt / 1000.0), "ms_step": ms_step, "ms_draft": ms_draft,
                    "ms_verify": ms_verify, "tau": tok / (nt * B),
                    "verify_roofline": {"frac": vbytes / ms_verify / 1e6 / peak,
                                        "achieved_gbs": vbytes / ms_verify / 1e6, "bytes": vbytes},
                    "draft_roofline": {"frac": dbytes / ms_draft / 1e6 / peak,
                                       "achieved_gbs": dbytes / ms_draft / 1e6, "bytes": dbytes},
                    "experts_touched_per_layer": touched, "peak_gbs": peak, "peak_source": peak_kind})
    eng.close()
    del eng
    torch.cuda.empty_cache()
    return out


def run_fp8_point(args, shape, vw, dw, ctx, pend, kvs, dkvs, dev, peak, peak_kind):
    """The bench step (draft + verify + commit, B=8, K=3, the same inputs) with the fp8-expert
    variant: expert matrices quantised to e4m3 with per-row scales (input construction on the
    host), e4m3 expert products.  Event pairs around each phase, per-step medians."""
    import torch

    import synth_inputs as S
    from paper_2609_03181_gb300 import fastmtp as F

    B, K = args.batch, args.K
    v8 = S.quantize_experts_fp8(vw)
    n_all = args.warmup + args.steps
    stream = torch.cuda.Stream(dev)
    eng = F.Engine(v8, dw, max_batch=B, K_max=K, max_ctx=max(ctx) + (n_all + 4) * (K + 1) + 8, page_size=64,
                   device=str(dev), stream=stream, expert_fp8=True)
    for b in range(B):
        eng.load_prefix(b, kvs[b], dkvs[b], pend[b])
    slots = torch.arange(B, dtype=torch.int32, device=dev)
    c0 = torch.tensor([[p] for p in pend], dtype=torch.int32, device=dev)
    v0 = torch.empty(B, 1, dtype=torch.int32, device=dev)
    acc = torch.empty(B, dtype=torch.int32, device=dev)
    cand = torch.empty(B, K + 1, dtype=torch.int32, device=dev)
    vt = torch.empty(B, K + 1, dtype=torch.int32, device=dev)
    com = torch.empty(B, K + 1, dtype=torch.int32, device=dev)
    hist = torch.zeros(n_all, B, dtype=torch.int32, device=dev)
    ev = [[torch.cuda.Event(enable_timing=True) for _ in range(4)] for _ in range(n_all)]
    torch.cuda.synchronize(dev)
    with torch.cuda.stream(stream):
        eng.verify_step(slots, c0, v0, acc)
        eng.accept_commit(slots, v0, acc)
        for i in range(n_all):
            if i == args.warmup:
                eng.profile(2)
            ev[i][0].record(stream)
            eng.draft_step(slots, K, cand)
            ev[i][1].record(stream)
            eng.verify_step(slots, cand, vt, acc)
            ev[i][2].record(stream)
            eng.accept_commit(slots, com, hist[i])
            ev[i][3].record(stream)
    eng.sync()
    counted = eng.profile_read()
    eng.close()
    del eng
    torch.cuda.empty_cache()
    timed = range(args.warmup, n_all)
    med = lambda a, b: statistics.median(ev[i][a].elapsed_time(ev[i][b]) for i in timed)
    ms_step, ms_verify = med(0, 3), med(1, 2)
    h = hist.double().cpu()
    tok = float(h[args.warmup:].sum())
    touched = counted["experts_touched"] / max(1, counted["launches"]["router"])
    ctx_mean = statistics.mean(ctx) + (args.warmup + args.steps / 2) * 2
    vbytes = algorithmic_bytes(shape, B, K, ctx_mean, touched - shape.n_shared, fp8_experts=True)
    return {"variant": "fp8 experts: e4m3 expert matrices with a per-row fp32 scale, e4m3 expert inputs and "
                       "activations (no counterpart in the paper)",
            "batch": B, "K": K, "steps": args.steps, "tokens_per_s": tok / (ms_step * args.steps / 1000.0),
            "ms_step": ms_step, "ms_verify": ms_verify, "ms_draft": med(0, 1), "tau": tok / (args.steps * B),
            "verify_roofline": {"frac": vbytes / ms_verify / 1e6 / peak, "achieved_gbs": vbytes / ms_verify / 1e6,
                                "bytes": vbytes, "peak_source": peak_kind}}


LOSS_ROWS, LOSS_K = 64, 3


def run_loss_point(args, shape, dev, peak, peak_kind, iters=20):
    """The draft-head objective (spec_draft_loss) over 64 rows and K = 3 depths with the full
    129,280-token LM head: W_lm (331 MB, larger than L2) streamed once per call.  CUDA events
    around `iters` back-to-back calls after 3 warm-up calls; roofline = max(bytes / HBM peak,
    FLOPs / bf16 peak) against the measured time."""
    import torch

    import synth_inputs as S
    from paper_2609_03181_gb300 import fastmtp as F

    R, K, V, d = LOSS_ROWS, LOSS_K, shape.vocab, shape.hidden
    u = S.normal(77, "loss.u", (K, R, d), 1.0).to(dev)
    b = S.normal(77, "loss.b", (R, d), 1.0).to(dev)
    W = S.normal(77, "loss.w", (V, d), 0.02).to(dev)
    tgt = torch.from_numpy(S.integers(77, "loss.t", R, 0, V - 1).astype("int32")).to(dev)
    ws = torch.empty(F.draft_loss_workspace_bytes(K, R, V), dtype=torch.uint8, device=dev)
    stream = torch.cuda.Stream(dev)
    torch.cuda.synchronize(dev)
    with torch.cuda.stream(stream):
        for _ in range(3):
            F.draft_loss(u, b, tgt, W, workspace=ws, stream=stream)
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        for _ in range(iters):
            out, _ = F.draft_loss(u, b, tgt, W, workspace=ws, stream=stream)
        e1.record(stream)
    torch.cuda.synchronize(dev)
    ms = e0.elapsed_time(e1) / iters
    rows_packed = R * 4
    byts = V * d * 2 + rows_packed * d * 2
    flops = 2.0 * V * d * rows_packed
    pk_tf = None
    try:
        pk_tf = float(json.load(open(os.path.join(ROOT, "MEASURED_PEAKS.json")))["bf16_tflops"])
    except Exception:
        pk_tf = 1900.0
    gbs = byts / ms / 1e6
    tfs = flops / ms / 1e9
    bound = "hbm" if byts / peak >= flops / (pk_tf * 1000.0) else "tensor"
    return {"rows": R, "K": K, "vocab": V, "ms": ms, "achieved_gbs": gbs, "hbm_frac": gbs / peak,
            "achieved_tflops": tfs, "tensor_frac": tfs / pk_tf, "bound": bound,
            "frac": max(gbs / peak, tfs / pk_tf), "algorithmic_bytes": byts, "flops": flops,
            "loss": float(out[0]), "peak_source": peak_kind,
            "timing": "CUDA events around back-to-back calls (pack, GEMM + softmax statistics, fold, mean)"}


def run_fastmtp(args):
    import torch
    import torch.distributed as dist

    from paper_2609_03181_gb300 import fastmtp as F

    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if world > 1:
        dist.init_process_group("nccl")
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)

    # the oracle sample runs first (rank 0, N=1 only), before any GPU work
    work = workload(args, rank)
    shape, vw, dw, ctx, pend, kvs, dkvs = work
    cpu_base = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        cpu_base = cpu_oracle_sample(args, work, args.cpu_budget_s)

    B, K = args.batch, args.K
    total_new = (args.warmup + args.steps) * (K + 1) * 2 + 2 * (K + 1) + 8
    stream = torch.cuda.Stream(dev)
    fp8 = args.experts == "fp8"
    eng = F.Engine(vw, dw, max_batch=B, K_max=K, max_ctx=max(ctx) + total_new, page_size=64, device=str(dev),
                   expert_fp8=fp8,
                   stream=stream)
    slots = torch.arange(B, dtype=torch.int32, device=dev)
    cand = torch.empty(B, K + 1, dtype=torch.int32, device=dev)
    vt = torch.empty(B, K + 1, dtype=torch.int32, device=dev)
    acc = torch.empty(B, dtype=torch.int32, device=dev)
    com = torch.empty(B, K + 1, dtype=torch.int32, device=dev)

    def reset():
        for b in range(B):
            eng.load_prefix(b, kvs[b], dkvs[b], pend[b])
        c0 = torch.tensor([[p] for p in pend], dtype=torch.int32, device=dev)
        v0 = torch.empty(B, 1, dtype=torch.int32, device=dev)
        torch.cuda.synchronize(dev)
        with torch.cuda.stream(stream):
            eng.verify_step(slots, c0, v0, acc)
            eng.accept_commit(slots, torch.empty(B, 1, dtype=torch.int32, device=dev), acc)
        eng.sync()

    def step(ncom_out):
        eng.draft_step(slots, K, cand)
        eng.verify_step(slots, cand, vt, acc)
        eng.accept_commit(slots, com, ncom_out)

    reset()
    ncom = torch.zeros(max(1, args.steps), B, dtype=torch.int32, device=dev)
    torch.cuda.synchronize(dev)
    with torch.cuda.stream(stream):
        for _ in range(args.warmup):
            step(ncom[0])
    eng.sync()

    # -------- timed region: device-resident inputs, CUDA-graph replays, CUDA events on the stream
    hist = torch.zeros(args.steps, B, dtype=torch.int32, device=dev)
    torch.cuda.synchronize(dev)
    ev = [torch.cuda.Event(enable_timing=True) for _ in range(2)]
    ph = [[torch.cuda.Event(enable_timing=True) for _ in range(4)] for _ in range(args.steps)]
    clocks = ClockSampler(local)
    eng.profile(2)                       # count launches and experts, no events
    if world > 1:
        dist.barrier()
    torch.cuda.synchronize(dev)
    clocks.start()
    with torch.cuda.stream(stream):
        ev[0].record(stream)
        for i in range(args.steps):
            ph[i][0].record(stream)
            eng.draft_step(slots, K, cand)
            ph[i][1].record(stream)
            eng.verify_step(slots, cand, vt, acc)
            ph[i][2].record(stream)
            eng.accept_commit(slots, com, hist[i])
            ph[i][3].record(stream)
        ev[1].record(stream)
    torch.cuda.synchronize(dev)
    clk = clocks.stop()
    if world > 1:
        dist.barrier()
    eng.sync()
    counted = eng.profile_read()
    # -------- the same steps again with an event pair around every launch group (per-kernel time)
    with torch.cuda.stream(stream):
        eng.profile(1)
        hist2 = torch.zeros(args.steps, B, dtype=torch.int32, device=dev)
        torch.cuda.synchronize(dev)
        for i in range(args.steps):
            step(hist2[i])
    eng.sync()
    prof = eng.profile_read()
    eng.profile(0)
    ms_total = ev[0].elapsed_time(ev[1])
    accepted = int(hist.sum().item())
    ms_draft = statistics.mean(ph[i][0].elapsed_time(ph[i][1]) for i in range(args.steps))
    ms_verify = statistics.mean(ph[i][1].elapsed_time(ph[i][2]) for i in range(args.steps))
    ms_commit = statistics.mean(ph[i][2].elapsed_time(ph[i][3]) for i in range(args.steps))
    m_hist = [0] * (K + 1)
    for n in hist.flatten().tolist():
        m_hist[n - 1] += 1
    ms_total, accepted_all = job_totals(ms_total, accepted, world, dev)
    value = accepted_all / (ms_total / 1000.0)

    # -------- e2e through the public API: pinned H2D of the step's input, D2H of its result
    e2e = None
    if not args.no_e2e:
        reset()
        h_slots = torch.arange(B, dtype=torch.int32).pin_memory()
        # two pinned result buffers: the host reads step i's result while step i+1 runs
        h_com = [torch.empty(B, K + 1, dtype=torch.int32).pin_memory() for _ in range(2)]
        h_n = [torch.empty(B, dtype=torch.int32).pin_memory() for _ in range(2)]
        done = [torch.cuda.Event() for _ in range(2)]
        d_n = torch.empty(B, dtype=torch.int32, device=dev)
        torch.cuda.synchronize(dev)
        with torch.cuda.stream(stream):
            for _ in range(args.warmup):
                step(d_n)
        eng.sync()
        if world > 1:
            dist.barrier()
        tok = 0
        t0 = time.perf_counter()
        with torch.cuda.stream(stream):
            for i in range(args.steps):
                slots.copy_(h_slots, non_blocking=True)
                step(d_n)
                h_com[i % 2].copy_(com, non_blocking=True)
                h_n[i % 2].copy_(d_n, non_blocking=True)
                done[i % 2].record(stream)
                if i > 0:
                    done[(i - 1) % 2].synchronize()
                    tok += int(h_n[(i - 1) % 2].sum())
            if args.steps > 0:
                last = (args.steps - 1) % 2
                done[last].synchronize()
                tok += int(h_n[last].sum())
        dt, tok = job_totals(time.perf_counter() - t0, tok, world, dev)
        e2e = {"value": tok / dt, "unit": "tokens/s", "h2d_bytes_per_step": B * 4,
               "d2h_bytes_per_step": B * (K + 1) * 4 + B * 4,
               "host_loop": ("every step: pinned H2D of the slots, the step, D2H of the committed tokens and "
                             "counts into one of two pinned buffers; the host reads step i's counts while "
                             "step i+1 runs")}
    eng.close()
    del eng
    torch.cuda.empty_cache()
    points = None
    loss_point = None
    fp8_point = None
    if not args.no_points and world == 1 and not fp8:
        pk, pkind = measured_peaks()
        points = run_points(args, shape, vw, dw, dev, pk, pkind)
        loss_point = run_loss_point(args, shape, dev, pk, pkind)
        if not fp8:
            fp8_point = run_fp8_point(args, shape, vw, dw, ctx, pend, kvs, dkvs, dev, pk, pkind)

    if rank != 0:
        if world > 1:
            dist.destroy_process_group()
        return

    # -------- roofline of the dominant kernel (live event timing) and of the verify step
    peak, peak_kind = measured_peaks()
    L = shape.n_layers
    steps = args.steps
    touched = counted["experts_touched"] / max(1, counted["launches"]["router"])     # per layer, incl. shared
    rows = counted["expert_rows"] / max(1, counted["launches"]["router"])
    d, I = shape.hidden, shape.expert_inter
    eb = 1 if fp8 else 2   # bytes per expert weight and per expert input / activation element
    sc = (4 * 2 * I, 4 * d) if fp8 else (0, 0)   # fp32 row scales of gate/up and down
    cls_bytes = {
        "expert_gate_up": touched * (2 * I * d * eb + sc[0]) + rows * d * eb + rows * I * eb,
        "expert_down": touched * (d * I * eb + sc[1]) + rows * I * eb + rows * d * 4,
        "lm_head": shape.vocab * d * 2.0,
    }
    fused = counted["launches"]["expert_down"] == 0   # gate/up and down run as one launch per layer
    if fused:
        cls_bytes["expert_gate_up"] += cls_bytes["expert_down"]
    gemm_ms = {k: prof["ms"][k] for k in ("expert_gate_up", "expert_down", "qkv", "oproj", "lm_head",
                                          "attention", "draft_gemm")}
    dom = max(("expert_gate_up", "expert_down", "lm_head"), key=lambda k: prof["ms"][k])
    dur_ms = prof["ms"][dom] / max(1, prof["launches"][dom])
    achieved = cls_bytes[dom] / (dur_ms / 1000.0) / 1e9
    label = "experts" if (fused and dom == "expert_gate_up") else dom
    traffic = None
    tpath = os.path.join(ROOT, "profiles", "ncu_traffic.json")
    if os.path.exists(tpath):
        tj = json.load(open(tpath))
        src = open(os.path.join(ROOT, "paper_2609_03181_gb300", "csrc", "gemm_tc.cu"), "rb").read()
        if tj.get("kernel_class") == label and tj.get("gemm_tc_sha256") == hashlib.sha256(src).hexdigest():
            traffic = tj.get("dram_bytes_per_launch")
    roofline = {"bound": "hbm", "achieved": achieved, "peak": peak, "unit": "GB/s", "frac": achieved / peak,
                "traffic": traffic, "kernel": label, "algorithmic_bytes_per_launch": cls_bytes[dom],
                "avg_launch_ms": dur_ms, "avg_launch_timing": "serialised replay (event pair per launch)",
                "peak_source": peak_kind}
    routed_touched = touched - shape.n_shared
    vbytes = algorithmic_bytes(shape, B, K, statistics.mean(ctx) + (args.warmup + steps / 2) * 2, routed_touched,
                               fp8_experts=fp8)
    v_ach = vbytes / (ms_verify / 1000.0) / 1e9
    ctx_run = statistics.mean(ctx) + (args.warmup + steps / 2) * 2
    dbytes = draft_algorithmic_bytes(shape, B, K, ctx_run, accepted / steps)
    d_ach = dbytes / (ms_draft / 1000.0) / 1e9
    launches_total = sum(counted["launches"].values())
    out = {
        "metric": METRIC, "value": value, "unit": "tokens/s", "n_gpus": world, "steps": steps,
        "warmup": args.warmup, "ms_per_step": ms_total / steps, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "bf16", "data": data_desc(args),
        "config": {"workload": WORKLOAD, "batch": B, "K": K, "layers": L, "ctx": f"U[{args.ctx_lo},{args.ctx_hi}]",
                   "weights": args.weights, "experts": args.experts,
                   "l2": "inputs larger than L2: 6.3 GB of weights streamed per step", "parallelism": "replicas"},
        "roofline": roofline,
        "verify_roofline": {"bound": "hbm", "achieved": v_ach, "peak": peak, "unit": "GB/s", "frac": v_ach / peak,
                            "algorithmic_bytes": vbytes, "ms": ms_verify},
        "draft_roofline": {"bound": "hbm", "achieved": d_ach, "peak": peak, "unit": "GB/s", "frac": d_ach / peak,
                           "algorithmic_bytes": dbytes, "ms": ms_draft},
        "phase_ms": {"draft": ms_draft, "verify": ms_verify, "commit": ms_commit},
        "kernel_ms_per_step": {k: v / steps for k, v in prof["ms"].items()},
        "kernel_ms_timing": ("serialised: a separate replay of the same steps with a CUDA event pair around "
                             "every launch group, which removes the programmatic-dependent-launch overlap "
                             "between kernels (sums exceed ms_per_step; roofline.avg_launch_ms is from it)"),
        "sweep_points": points,
        "draft_objective": loss_point,
        "fp8_experts": fp8_point,
        "tau": accepted / (steps * B), "accept_hist_m": m_hist,
        "experts_touched_per_layer": touched,
        "gpu_launches": launches_total,
        "clocks": clk,
        "e2e": e2e,
        "cpu_baseline": cpu_base,
    }
    print(json.dumps(out), flush=True)
    if world > 1:
        dist.destroy_process_group()


# ----------------------------------------------------------------------------- sweep
def run_sweep(args):
    """Every (router, context, batch, K) point of the grid on one engine per router mode:
    committed contexts of exactly `ctx` tokens (N(0,1) KV drawn on the device), one K=0 step
    to seed the draft head, `warmup` steps, then `steps` timed steps with an event pair around
    each phase (medians over the timed steps).  Weights: the acceptance-tuned seeded set
    (seed 4); the Zipf mode adds the per-expert router bias -1.2 ln(rank).  Pending tokens use
    seeds 4..8 by batch size."""
    import torch

    import synth_inputs as S
    from paper_2609_03181_gb300 import fastmtp as F
    from paper_2609_03181_gb300 import metrics as M

    batches = [int(x) for x in args.sweep_batch.split(",")]
    ctxs = [int(x) for x in args.sweep_ctx.split(",")]
    Ks = [int(x) for x in args.sweep_k.split(",")]
    routers = args.sweep_router.split(",")
    dev = torch.device("cuda", 0)
    torch.cuda.set_device(dev)
    peak, peak_kind = measured_peaks()
    shape = S.ModelShape(n_layers=args.layers)
    Bmax, Kmax = max(batches), max(Ks)
    steps_for = lambda B: max(args.steps, 50) if B <= 4 else args.steps   # acceptance varies most at small B
    grow = (args.warmup + steps_for(1) + 2) * (Kmax + 1)
    clocks = ClockSampler(0)
    clocks.start()
    fp8 = args.experts == "fp8"
    for router in routers:
        vw, dw, _ = S.successor_weights(shape, 4, ACCEPT_RATIO)
        if router == "zipf":
            for l, lw in enumerate(vw.layers):
                lw.router_bias = S.zipf_router_bias(4, l, shape.n_experts, 1.2)
        if fp8:
            vw = S.quantize_experts_fp8(vw)
        stream = torch.cuda.Stream(dev)
        eng = F.Engine(vw, dw, max_batch=Bmax, K_max=Kmax, max_ctx=max(ctxs) + grow, page_size=64,
                       device=str(dev), stream=stream, expert_fp8=fp8)
        g = torch.Generator(device=dev)
        g.manual_seed(4)
        for l in range(shape.n_layers):
            eng.kv_pool[l].normal_(generator=g)
        eng.dkv_pool.normal_(generator=g)
        # tensors made on PyTorch's current stream are complete before the engine's stream reads them
        torch.cuda.synchronize(dev)
        for ctx in ctxs:
            for bi, B in enumerate(batches):
                pend = [int(t) for t in S.integers(4 + bi, "pending", B, 0, shape.vocab - 1)]
                slots = torch.arange(B, dtype=torch.int32, device=dev)
                c0 = torch.tensor([[p] for p in pend], dtype=torch.int32, device=dev)
                v0 = torch.empty(B, 1, dtype=torch.int32, device=dev)
                ar_tok_s = None   # greedy autoregressive (K=0) throughput of this (router, ctx, B)
                n_steps = steps_for(B)
                by_k = {}
                for K in Ks:
                    for b in range(B):
                        eng.reset_seq(b, ctx, eng.block_table(b), pend[b])
                    acc = torch.empty(B, dtype=torch.int32, device=dev)
                    cand = torch.empty(B, K + 1, dtype=torch.int32, device=dev)
                    vt = torch.empty(B, K + 1, dtype=torch.int32, device=dev)
                    com = torch.empty(B, K + 1, dtype=torch.int32, device=dev)
                    n_all = args.warmup + n_steps
                    hist = torch.zeros(n_all, B, dtype=torch.int32, device=dev)
                    ev = [[torch.cuda.Event(enable_timing=True) for _ in range(4)] for _ in range(n_all)]
                    torch.cuda.synchronize(dev)
                    with torch.cuda.stream(stream):
                        eng.verify_step(slots, c0, v0, acc)
                        eng.accept_commit(slots, v0, acc)
                    eng.sync()
                    # K=0 is plain greedy decoding: no draft step; each verify takes the token the
                    # previous commit wrote (two buffers, alternating)
                    ar_bufs = [v0, torch.empty_like(v0)]
                    with torch.cuda.stream(stream):
                        for i in range(n_all):
                            if i == args.warmup:
                                eng.profile(2)
                            ev[i][0].record(stream)
                            if K > 0:
                                eng.draft_step(slots, K, cand)
                            ev[i][1].record(stream)
                            eng.verify_step(slots, cand if K > 0 else ar_bufs[i % 2], vt, acc)
                            ev[i][2].record(stream)
                            eng.accept_commit(slots, com if K > 0 else ar_bufs[(i + 1) % 2], hist[i])
                            ev[i][3].record(stream)
                    eng.sync()
                    counted = eng.profile_read()
                    eng.profile(0)
                    cnt = eng.read_workspace(F.WS_EXPERT_CNT, (shape.n_layers, shape.n_experts), torch.int32).double()
                    timed = range(args.warmup, n_all)
                    # medians over the timed steps: a host stall between two launches shows up
                    # in one step's event pair and would skew a mean
                    ms = lambda a, b: statistics.median(ev[i][a].elapsed_time(ev[i][b]) for i in timed)
                    ms_step, ms_draft, ms_verify = ms(0, 3), ms(0, 1), ms(1, 2)
                    h = hist.double().cpu()
                    lens = ctx + 1 + torch.cumsum(h, 0) - h          # committed length seen by each verify
                    ctx_mean = float(lens[args.warmup:].mean())
                    tok = float(h[args.warmup:].sum())
                    touched = counted["experts_touched"] / max(1, counted["launches"]["router"])
                    vbytes = algorithmic_bytes(shape, B, K, ctx_mean, touched - shape.n_shared, fp8)
                    load = cnt / cnt.mean(-1, keepdim=True)
                    tok_s = tok / (ms_step * n_steps / 1000.0)
                    if K == 0:
                        ar_tok_s = tok_s
                    out = {"sweep": True, "router": router, "experts": args.experts, "batch": B, "ctx": ctx, "K": K,
                           "tokens_per_s": tok_s, "ms_step": ms_step,
                           "ms_step_mean": statistics.mean(ev[i][0].elapsed_time(ev[i][3]) for i in timed),
                           "ms_draft": ms_draft, "ms_verify": ms_verify, "ms_commit": ms(2, 3),
                           "tau": tok / (n_steps * B),
                           "verify_roofline": {"bytes": vbytes, "achieved_gbs": vbytes / ms_verify / 1e6,
                                               "peak": peak, "peak_source": peak_kind,
                                               "frac": vbytes / ms_verify / 1e6 / peak},
                           "experts_touched_per_layer": touched,
                           "expert_load_max_over_mean": float(load.max(-1).values.mean()),
                           "expert_share_top1": float((cnt.max(-1).values / cnt.sum(-1)).mean()),
                           "steps": n_steps, "warmup": args.warmup}
                    if ar_tok_s is not None:
                        # the paper's speedup over greedy decoding and step cost c = tau / S
                        sp = M.speedup_vs_ar(tok_s, ar_tok_s, out["tau"])
                        out["speedup_vs_ar"], out["step_cost_c"] = sp["S"], sp["c"]
                    print(json.dumps(out), flush=True)
                    by_k[K] = tok_s
                if 0 in by_k:
                    # the depth the packaged table's policy picks for this point, beside the best
                    # depth measured here
                    best = M.best_depth(by_k)
                    print(json.dumps({"sweep_best": True, "router": router, "batch": B, "ctx": ctx,
                                      "K_best_measured": best["k"], "S_best": best["S"],
                                      "K_policy": F.choose_depth(B, ctx)}), flush=True)
        eng.close()
        del eng
        torch.cuda.empty_cache()
    clk = clocks.stop()
    print(json.dumps({"sweep_clocks": clk}), flush=True)


def run_trace(args):
    """One graph-replayed step (draft + verify + commit) of the bench workload, traced per CTA by
    the FASTMTP_TRACE=1 build of the library (entry, wait return and exit times).  Not a timing
    run: the records add a few atomics and stores per CTA.  Prints every launch, then the mean
    verify-layer breakdown (ready -> done per kernel and the hand-over gaps), as JSON lines."""
    os.environ["FASTMTP_TRACE"] = "1"   # read when the build module is first imported
    import torch

    from paper_2609_03181_gb300 import fastmtp as F
    from paper_2609_03181_gb300 import trace as TR

    dev = torch.device("cuda", 0)
    torch.cuda.set_device(dev)
    shape, vw, dw, ctx, pend, kvs, dkvs = workload(args, 0)
    B, K = args.batch, args.K
    stream = torch.cuda.Stream(dev)
    eng = F.Engine(vw, dw, max_batch=B, K_max=K, max_ctx=max(ctx) + (args.warmup + 4) * (K + 1) + 8, page_size=64,
                   device=str(dev), stream=stream, expert_fp8=args.experts == "fp8")
    slots = torch.arange(B, dtype=torch.int32, device=dev)
    cand = torch.empty(B, K + 1, dtype=torch.int32, device=dev)
    vt = torch.empty(B, K + 1, dtype=torch.int32, device=dev)
    acc = torch.empty(B, dtype=torch.int32, device=dev)
    com = torch.empty(B, K + 1, dtype=torch.int32, device=dev)
    ncom = torch.empty(B, dtype=torch.int32, device=dev)
    for b in range(B):
        eng.load_prefix(b, kvs[b], dkvs[b], pend[b])
    c0 = torch.tensor([[p] for p in pend], dtype=torch.int32, device=dev)
    v0 = torch.empty(B, 1, dtype=torch.int32, device=dev)
    torch.cuda.synchronize(dev)

    def step():
        eng.draft_step(slots, K, cand)
        eng.verify_step(slots, cand, vt, acc)
        eng.accept_commit(slots, com, ncom)

    with torch.cuda.stream(stream):
        eng.verify_step(slots, c0, v0, acc)
        eng.accept_commit(slots, v0, acc)
        for _ in range(max(1, args.warmup)):
            step()
    eng.sync()
    F.trace_read(reset=True)   # drop the warm-up records
    with torch.cuda.stream(stream):
        step()
    eng.sync()
    recs = F.trace_read(reset=True)
    if args.trace_out:
        import numpy as np
        np.save(args.trace_out, recs)
    ls = TR.launches(recs)
    for g in ls:
        print(json.dumps({"launch": g["name"], "kid": g["kid"], "grid": [g["grid_x"], g["grid_y"]], "ctas": g["ctas"],
                          "entry_us": g["entry"], "ready_us": g["ready"], "done_us": g["done"]}), flush=True)
    layers = TR.verify_layers(ls)
    print(json.dumps({"trace": True, "batch": B, "K": K, "ctx": [args.ctx_lo, args.ctx_hi], "layers": args.layers,
                      "experts": args.experts, "records": int(len(recs)), "launches": len(ls), "verify_layers": len(layers),
                      "verify_layer_us": TR.layer_breakdown(layers)}), flush=True)
    eng.close()


def main():
    args = parse()
    if args.trace:
        run_trace(args)
        return
    if args.objective:
        import torch
        import synth_inputs as S
        torch.cuda.set_device(0)
        pk, pkind = measured_peaks()
        print(json.dumps({"draft_objective": run_loss_point(args, S.ModelShape(), torch.device("cuda", 0), pk, pkind)}),
              flush=True)
        return
    if args.sweep:
        run_sweep(args)
    elif args.impl == "reference":
        run_reference(args)
    else:
        run_fastmtp(args)


if __name__ == "__main__":
    main()
