"""Host-side grouping of the device timeline (paper_2609_03181_gb300/trace.py) on synthetic
records laid out as spec_trace_read returns them; no GPU needed."""
import numpy as np

from paper_2609_03181_gb300 import trace as TR


def sig(kid, grid, block, exit_=False):
    return (kid << 48) | (grid << 32) | (1 << 16) | block | ((1 << 63) if exit_ else 0)


def launch(recs, kid, grid, block, t_entry, t_ready, t_exit=None, ctas=3):
    for c in range(ctas):
        recs.append([sig(kid, grid, block), c, t_entry + 100 * c, t_ready + 50 * c])
        if t_exit is not None:
            recs.append([sig(kid, grid, block, True), c, t_exit + 200 * c, 0])


def two_layers():
    recs, t = [], 1_000_000
    launch(recs, 19, 4, 128, t, t + 500)                       # embedding (no exit records)
    for layer in range(2):
        base = t + 2_000 + layer * 100_000
        for j, kid in enumerate(TR.VERIFY_LAYER):
            launch(recs, kid, 80 + j, 192, base + 10_000 * j - 5_000, base + 10_000 * j, base + 10_000 * j + 6_000)
    launch(recs, 6, 152, 192, t + 300_000, t + 301_000, t + 350_000)   # LM head
    return np.array(recs, dtype=np.uint64)


def test_launches_group_ctas_and_order_by_ready_time():
    ls = TR.launches(two_layers())
    assert [g["name"] for g in ls][:7] == ["embed", "gemm_qkv", "attention", "gemm_resid", "router", "experts", "combine"]
    assert len(ls) == 1 + 2 * 6 + 1
    assert all(g["ctas"] == 3 for g in ls)
    q = ls[1]
    # microseconds from the first entry of the trace (layer 0's QKV enters 3 us before t)
    assert q["ready"] == (5.0, 5.1) and q["entry"] == (0.0, 0.2)
    assert q["done"] == (11.0, 11.4)                                  # its own exit records only
    assert ls[0].get("done_from_next") and ls[0]["done"] == (ls[1]["ready"][0],) * 2


def test_verify_layers_and_breakdown():
    ls = TR.launches(two_layers())
    layers = TR.verify_layers(ls)
    assert len(layers) == 2 and all([g["kid"] for g in L] == list(TR.VERIFY_LAYER) for L in layers)
    b = TR.layer_breakdown(layers)
    # every kernel: ready -> last exit = 6.0 + 0.4 us; hand-over from the previous kernel's last
    # exit (ready 10 us later, minus 6.4) = 3.6 us; layer 2 starts 100 us after layer 1
    assert abs(b["gemm_qkv"] - 6.4) < 1e-9 and abs(b["experts"] - 6.4) < 1e-9
    assert abs(b["gap_before_attention"] - 3.6) < 1e-9
    assert abs(b["gap_before_gemm_qkv"] - (100.0 - 50.0 - 6.4)) < 1e-9
    assert abs(b["layer"] - 56.4) < 1e-9


def test_launch_in_two_waves_stays_one_launch():
    # 152 CTAs enter at once, 104 more only as the first ones leave (their waits return at entry,
    # far from the first wave's); a second kernel enters after the last of them
    recs = []
    for c in range(256):
        t_in = 1_000 if c < 152 else 20_000 + 100 * c
        recs.append([sig(17, 256, 256), c, t_in, max(t_in, 5_000)])
    for c in range(4):
        recs.append([sig(7, 152, 192), c, 60_000 + c, 61_000])
    ls = TR.launches(np.array(recs, dtype=np.uint64))
    assert [(g["name"], g["ctas"]) for g in ls] == [("router", 256), ("experts", 4)]


def test_same_kernel_split_only_by_another_kernels_entry():
    recs = []
    for c in range(3):
        recs.append([sig(20, 3, 128), c, 1_000 + c, 2_000])        # RMSNorm launch 1
    recs.append([sig(1, 10, 192), 0, 2_500, 3_000])                # a GEMM in between
    for c in range(3):
        recs.append([sig(20, 3, 128), c, 2_600 + c, 4_000])        # RMSNorm launch 2, 1.6 us later
    ls = TR.launches(np.array(recs, dtype=np.uint64))
    assert [(g["name"], g["ctas"]) for g in ls] == [("rmsnorm", 3), ("gemm_f32", 1), ("rmsnorm", 3)]


def test_empty_trace():
    assert TR.launches(np.zeros((0, 4), dtype=np.uint64)) == []
    assert TR.verify_layers([]) == []
