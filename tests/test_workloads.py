"""The workload presets (synth_inputs.CONFIGS) and bench.py's defaults agree: the bench's step
is cfg1 and its sweep grid cfg4."""
import sys

import synth_inputs as S


def test_bench_defaults_are_cfg1_and_cfg4(monkeypatch):
    monkeypatch.setattr(sys, "argv", ["bench.py"])
    import bench
    a = bench.parse()
    c1, c4 = S.CONFIGS["cfg1"], S.CONFIGS["cfg4"]
    assert (a.batch, a.K, a.ctx_lo, a.ctx_hi, a.layers, a.seed) == (c1.batch, c1.K, c1.ctx_lo, c1.ctx_hi,
                                                                   c1.n_layers, c1.seed)
    assert [int(x) for x in a.sweep_batch.split(",")] == list(c4.grid["batch"])
    assert [int(x) for x in a.sweep_ctx.split(",")] == list(c4.grid["ctx"])
    assert [int(x) for x in a.sweep_k.split(",")] == list(c4.grid["K"])
    assert a.sweep_router.split(",") == list(c4.grid["router"])


def test_presets_are_consistent():
    assert sorted(S.CONFIGS) == ["cfg0", "cfg1", "cfg2", "cfg3", "cfg4"]
    for name, w in S.CONFIGS.items():
        assert 1 <= w.batch <= 256 and 1 <= w.K <= 7 and 1 <= w.ctx_lo <= w.ctx_hi
        assert w.ctx_hi + w.K + 1 <= S.ModelShape().max_position
        assert w.draft_only == (w.n_layers == 0)
    assert S.CONFIGS["cfg4"].grid["K"][0] == 0          # the greedy baseline of the speedup
    assert S.CONFIGS["cfg3"].gen_tokens == 512
