"""Host-side logic of the per-operator threshold calibration (no GPU)."""
import json
import math
import os

import numpy as np
import pytest
import torch

from paper_2511_19457_gb300 import calibrate as cal
from paper_2511_19457_gb300 import synth


def test_crossover_rules():
    r = [0.0, 0.3, 0.5, 0.7, 0.9]
    # zero-skip faster from 0.5 on
    assert cal.crossover(r, [10, 10, 10, 10, 10], [12, 11, 9, 8, 5]) == 0.5
    # never faster
    assert cal.crossover(r, [10] * 5, [11] * 5) == cal.NEVER
    # faster everywhere: zero-skip even on dense input
    assert cal.crossover(r, [10] * 5, [9] * 5) == 0.0
    # a win that does not last to the top of the grid does not count
    assert cal.crossover(r, [10] * 5, [12, 9, 11, 8, 7]) == 0.7
    # a tie is not a win
    assert cal.crossover(r, [10] * 5, [12, 11, 10, 9, 9]) == 0.7
    assert cal.crossover(r, [10] * 5, [12, 11, 9, 9, 10]) == cal.NEVER


def test_never_threshold_is_never_met():
    # the dispatch rule: zero-skip iff zeros >= s_thr * numel; zeros <= numel
    for numel in (1, 7, 1 << 20):
        assert not numel >= cal.NEVER * numel


def test_kinds():
    assert cal.kind_of("fc", (8, 512, 1000)) == "fc_small"
    assert cal.kind_of("fc", (128, 512, 1000)) == "fc_small"
    assert cal.kind_of("fc", (129, 512, 1000)) == "gemm"
    assert cal.kind_of("conv", (8, 56, 56, 64, 64, 3, 1, 1)) == "conv3x3s1"
    assert cal.kind_of("conv", (8, 56, 56, 64, 128, 1, 2, 0)) == "conv1x1s2"


def _brute_macs_conv(B, H, W, C, Co, k, s, p):
    """MACs counted output by output, tap by tap (taps in the padding still count)."""
    Ho = len(range(-p, H + p - k + 1, s))
    Wo = len(range(-p, W + p - k + 1, s))
    return B * Ho * Wo * Co * C * k * k


@pytest.mark.parametrize("shape", [(2, 7, 9, 8, 16, 3, 1, 1), (1, 8, 8, 16, 8, 3, 2, 1),
                                   (3, 5, 6, 8, 8, 1, 2, 0), (1, 224, 224, 3, 64, 7, 2, 3)])
def test_conv_flops_brute(shape):
    assert cal.flops_of("conv", shape) == 2 * _brute_macs_conv(*shape)


def test_resnet18_flops_table2():
    """ResNet-18 is quoted at 1.8 GMACs per 224x224 image (Table 2); the sum
    over the graph's convs and FC from the propagated shapes lands there."""
    ops, _, shape = synth.resnet18(batch=1)
    ins = cal.graph_input_shapes(ops, shape)
    macs = 0.0
    for op, (B, H, W, C) in zip(ops, ins):
        if op["kind"] == "conv":
            macs += cal.flops_of("conv", (B, H, W, C, op["cout"], op["k"], op["stride"], op["pad"])) / 2
        elif op["kind"] == "fc":
            macs += cal.flops_of("fc", (B, H * W * C, op["cout"])) / 2
    assert 1.75e9 < macs < 1.85e9


def test_graph_input_shapes_resnet18():
    ops, _, shape = synth.resnet18(batch=2)
    ins = cal.graph_input_shapes(ops, shape)
    assert ins[0] == (2, 224, 224, 3)
    assert ins[1] == (2, 112, 112, 64)          # max pool after the 7x7/2 stem
    assert ins[2] == (2, 56, 56, 64)
    assert ins[-2] == (2, 7, 7, 512)            # global average pool
    assert ins[-1] == (2, 1, 1, 512)            # FC
    # each conv's input channel count is what the op expects
    for op, s in zip(ops, ins):
        if op["kind"] == "conv":
            assert s[3] == op["cin"]


def test_graph_input_shapes_mobilenet_v2():
    ops, _, shape = synth.mobilenet_v2(batch=1)
    ins = cal.graph_input_shapes(ops, shape)
    for op, s in zip(ops, ins):
        if op["kind"] in ("conv", "fc"):
            assert s[1] * s[2] * s[3] == op["cin"] or s[3] == op["cin"]
    assert ins[-1] == (1, 1, 1, 1280)


def _table():
    e = lambda kind, gf, s, st="unstructured": {"kind": kind, "structure": st, "flops": gf * 1e9, "s_thr": s}
    return {"entries": [e("conv3x3s1", 1.0, 0.6), e("conv3x3s1", 10.0, cal.NEVER),
                        e("conv3x3s1", 1.0, 0.3, "block"), e("fc_small", 0.01, 0.0),
                        e("conv1x1s2", 0.1, 0.8)]}


def test_thresholds_nearest_in_log_flops():
    t = _table()
    small = (8, 56, 56, 64, 64, 3, 1, 1)   # 3.7 GFLOP: nearer 1 than 10 in log
    big = (32, 56, 56, 64, 64, 3, 1, 1)    # 14.8 GFLOP
    assert cal.thresholds_for(t, "conv", small) == {"s_thr": 0.6, "c_thr": 0.0}
    assert cal.thresholds_for(t, "conv", big)["s_thr"] == cal.NEVER
    assert cal.thresholds_for(t, "conv", small, "block")["s_thr"] == 0.3
    assert cal.thresholds_for(t, "conv", (8, 56, 56, 64, 128, 3, 2, 1)) is None  # kind absent
    assert cal.thresholds_for(t, "fc", (8, 512, 1000))["s_thr"] == 0.0
    assert cal.thresholds_for(t, "fc", (4096, 512, 1000)) is None  # gemm kind absent


def test_apply_leaves_stem_depthwise_and_unknown_kinds():
    ops, _, shape = synth.mobilenet_v2(batch=1)
    out = cal.apply(ops, shape, {"entries": [
        {"kind": "conv1x1s1", "structure": "unstructured", "flops": 1e8, "s_thr": 0.7},
        {"kind": "conv3x3s2", "structure": "unstructured", "flops": 1e8, "s_thr": 0.1},
        {"kind": "fc_small", "structure": "unstructured", "flops": 1e6, "s_thr": 0.0}]})
    assert len(out) == len(ops)
    for a, b in zip(ops, out):
        if b["kind"] == "conv" and b["groups"] == 1 and b["k"] == 1:
            assert b["thr"] == {"s_thr": 0.7, "c_thr": 0.0}
        elif b["kind"] == "fc":
            assert b["thr"] == {"s_thr": 0.0, "c_thr": 0.0}
        else:  # the stem (on the graph input), depthwise, pools
            assert b.get("thr", {}) == a.get("thr", {})
    assert ops[0].get("thr") == {}  # the input list is not modified


def test_structured_activation_block_units():
    g = torch.Generator().manual_seed(1)
    x = synth.structured_activation((300, 100), 0.5, "block", g).float()
    z = (x == 0)
    for r0 in range(0, 300, 128):
        for c0 in range(0, 100, 32):
            u = z[r0:r0 + 128, c0:c0 + 32]
            assert bool(u.all()) or not bool(u.any())
    y = synth.structured_activation((2, 20, 9, 70), 0.5, "block", g).float()
    zy = (y == 0)
    for b in range(2):
        for h0 in range(0, 20, 8):
            for c0 in range(0, 70, 64):
                u = zy[b, h0:h0 + 8, :, c0:c0 + 64]
                assert bool(u.all()) or not bool(u.any())
    big = synth.structured_activation((512, 4096), 0.7, "unstructured", g).float()
    assert abs(float((big == 0).float().mean()) - 0.7) < 0.01
    assert float(big[big != 0].min()) >= 1e-3 * 0.99


def test_committed_table_is_consistent():
    if not os.path.exists(cal.TABLE_PATH):
        pytest.skip("no calibration table committed")
    t = cal.load_table()
    assert t["entries"]
    for e in t["entries"]:
        assert e["kind"] == cal.kind_of(e["op"], e["shape"])
        assert math.isclose(e["flops"], cal.flops_of(e["op"], e["shape"]))
        assert e["s_thr"] == cal.crossover(e["rho"], e["dense_us"], e["skip_us"])
        assert all(v > 0 for v in e["dense_us"] + e["skip_us"])
