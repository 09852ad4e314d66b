"""The workload presets (synth_inputs.WORKLOADS) and bench.py's defaults agree: the bench's
step is the 12-layer B=8 verify workload and its sweep grid the sweep workload's axes."""
import sys

import synth_inputs as S

STEP, SWEEP = "verify_12l_b8_ctx768_1024", "sweep_12l_b1_256_ctx1024_8192"


def test_bench_defaults_are_the_step_and_sweep_workloads(monkeypatch):
    monkeypatch.setattr(sys, "argv", ["bench.py"])
    import bench
    a = bench.parse()
    st, sw = S.WORKLOADS[STEP], S.WORKLOADS[SWEEP]
    assert (a.batch, a.K, a.ctx_lo, a.ctx_hi, a.layers, a.seed) == (st.batch, st.K, st.ctx_lo, st.ctx_hi,
                                                                   st.n_layers, st.seed)
    assert [int(x) for x in a.sweep_batch.split(",")] == list(sw.grid["batch"])
    assert [int(x) for x in a.sweep_ctx.split(",")] == list(sw.grid["ctx"])
    assert [int(x) for x in a.sweep_k.split(",")] == list(sw.grid["K"])
    assert a.sweep_router.split(",") == list(sw.grid["router"])


def test_presets_are_consistent():
    assert len(S.WORKLOADS) == 5
    for name, w in S.WORKLOADS.items():
        assert 1 <= w.batch <= 256 and 1 <= w.K <= 7 and 1 <= w.ctx_lo <= w.ctx_hi
        assert w.ctx_hi + w.K + 1 <= S.ModelShape().max_position
        assert w.draft_only == (w.n_layers == 0)
        # the name carries the batch and the context range
        assert f"_b{w.batch}_" in name or f"_b1_{w.batch}_" in name, name
        assert f"ctx{w.ctx_lo}" in name, name
    assert S.WORKLOADS[SWEEP].grid["K"][0] == 0          # the greedy baseline of the speedup
    assert S.WORKLOADS["loop_12l_b64_ctx1024_4096"].gen_tokens == 512


def test_verify_bytes_match_the_derived_roofline_table():
    """bench.algorithmic_bytes (the numerator of every verify roofline fraction) against byte
    counts worked out by hand from the model's shapes (K=3; routed experts touched per layer
    under uniform routing, 64 (1 - (58/64)^T)): 2.44 GB at B=1, ctx 1024 (20.8 experts); 6.15 GB
    at B=8, ctx ~896 (61.3); 22.1 GB at B=64, ctx 4096 (64); 134.9 GB at B=256, ctx 8192 (64),
    each to three digits."""
    import bench
    sh = S.ModelShape()
    for B, ctx, experts, gb in ((1, 1024, 20.8, 2.44), (8, 896, 61.3, 6.15), (64, 4096, 64, 22.1),
                                (256, 8192, 64, 134.9)):
        got = bench.algorithmic_bytes(sh, B, 3, ctx, experts) / 1e9
        assert abs(got - gb) <= 0.006 * gb, (B, got, gb)
