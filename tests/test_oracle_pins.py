"""Pins of the oracle to things other than itself (CPU only).

Each check ties an oracle function to brute force on tiny inputs, a library
routine (torch float64 conv/pool, numpy matmul), a closed form, or a figure
printed in the SparOA paper (tests/golden/), so that a dropped term, a wrong
sign or index, or a transposed operand in the oracle fails here.
"""
import bisect
import math
import os
from fractions import Fraction

import numpy as np
import pytest
import torch
import torch.nn.functional as F

from oracle import oracle as orc
from paper_2511_19457_gb300 import synth

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _golden(name):
    out = {}
    with open(os.path.join(GOLDEN, name)) as f:
        for line in f:
            line = line.strip()
            if line and not line.startswith("#"):
                k, v = line.split("=", 1)
                out[k] = v
    return out


def _rand_bits(shape, rng, zero_p=0.5, specials=True):
    """bf16 bit patterns: N(0,1) values, a zero_p share of +0/-0, and (optionally)
    a few subnormals, infinities and NaNs."""
    v = rng.standard_normal(shape).astype(np.float32)
    bits = synth.to_bf16_bits(torch.from_numpy(v))
    z = rng.random(shape) < zero_p
    neg = rng.random(shape) < 0.5
    bits[z & neg] = 0x8000
    bits[z & ~neg] = 0x0000
    if specials and bits.size > 20:
        flat = bits.reshape(-1)
        idx = rng.choice(flat.size, size=6, replace=False)
        flat[idx] = [0x0001, 0x8003, 0x007F, 0x7F80, 0xFF80, 0x7FC1]
    return bits


# ---------------------------------------------------------------------------
# bf16 conversion
# ---------------------------------------------------------------------------
def test_bf16_to_f64_is_upper_half_of_binary32():
    allbits = np.arange(65536, dtype=np.uint32).astype(np.uint16)
    got = orc.bf16_to_f64(allbits)
    ref = (allbits.astype(np.uint32) << 16).view(np.float32).astype(np.float64)
    nan = np.isnan(ref)
    assert np.array_equal(np.isnan(got), nan)
    assert np.array_equal(got[~nan], ref[~nan])
    # signs of the zeros survive
    assert math.copysign(1.0, got[0x8000]) == -1.0 and math.copysign(1.0, got[0]) == 1.0


def _finite_bf16_sorted():
    vals = []
    for b in range(65536):
        e = (b >> 7) & 0xFF
        if e == 0xFF:
            continue
        f = b & 0x7F
        mag = Fraction(f, 2 ** 133) if e == 0 else Fraction(128 + f, 1) * Fraction(2) ** (e - 134)
        vals.append((-mag if b >> 15 else mag, b))
    vals.sort(key=lambda t: t[0])
    return vals


def _rne_bruteforce(x: float, table):
    """Nearest finite bf16 by exact rational comparison, ties to even fraction;
    beyond the largest finite value by half an ulp or more -> infinity."""
    fx = Fraction(x)
    keys = [t[0] for t in table]
    i = bisect.bisect_left(keys, fx)
    cands = [table[j] for j in (i - 1, i) if 0 <= j < len(table)]
    maxf = Fraction(255, 1) * Fraction(2) ** 120   # (2 - 2^-7) * 2^127
    half_ulp_top = Fraction(2) ** (127 - 8)
    if fx >= maxf + half_ulp_top:
        return 0x7F80
    if fx <= -(maxf + half_ulp_top):
        return 0xFF80
    best = min(cands, key=lambda t: (abs(t[0] - fx), t[1] & 1))
    if best[0] == 0:   # keep the sign of the input on a zero result
        return 0x8000 if math.copysign(1.0, x) < 0 else 0x0000
    return best[1]


def test_f64_to_bf16_round_to_nearest_even_bruteforce():
    table = _finite_bf16_sorted()
    rng = np.random.default_rng(1)
    xs = list(rng.standard_normal(300) * 10.0 ** rng.integers(-45, 38, 300))
    # exact midpoints between neighbours (ties) and points just off them
    for b in [0x3F80, 0x3F81, 0x4000, 0x0001, 0x0080, 0x7F7E, 0x8081, 0x0000]:
        lo = orc.bf16_to_f64(np.array([b], dtype=np.uint16))[0]
        hi = orc.bf16_to_f64(np.array([b + 1], dtype=np.uint16))[0]
        mid = (lo + hi) / 2.0
        xs += [mid, math.nextafter(mid, math.inf), math.nextafter(mid, -math.inf), -mid]
    # double-rounding trap: just above a tie by less than a binary32 ulp
    xs += [1.0 + 2.0 ** -8 + 2.0 ** -40, 1.0 + 2.0 ** -8 - 2.0 ** -40]
    # overflow boundary and deep subnormals
    xs += [3.3895313892515355e38, 3.40e38, 3.3961775292304135e38, 1e-45, 5e-324, -5e-324]
    got = orc.f64_to_bf16(np.array(xs, dtype=np.float64))
    for x, g in zip(xs, got):
        assert int(g) == _rne_bruteforce(float(x), table), (x, hex(int(g)))


def test_f64_to_bf16_matches_torch_for_binary32_inputs():
    rng = np.random.default_rng(2)
    v = (rng.standard_normal(200000) * 10.0 ** rng.integers(-40, 38, 200000)).astype(np.float32)
    v[:4] = [0.0, -0.0, np.inf, -np.inf]
    ref = synth.to_bf16_bits(torch.from_numpy(v))
    got = orc.f64_to_bf16(v.astype(np.float64))
    assert np.array_equal(got, ref)
    assert int(orc.f64_to_bf16(np.array([np.nan]))[0]) & 0x7FFF > 0x7F80


# ---------------------------------------------------------------------------
# Eq. 1 statistics and bitmaps: brute force
# ---------------------------------------------------------------------------
def _brute_stats(bits, R, C):
    vals = (bits.astype(np.uint32) << 16).view(np.float32).reshape(R, C)
    nz = [[(not (vals[r, c] == 0.0)) for c in range(C)] for r in range(R)]
    T = (C + 63) // 64
    W64 = (T + 63) // 64
    RB = (R + 127) // 128
    C32 = (C + 31) // 32
    nnz = sum(sum(row) for row in nz)
    col = [sum(nz[r][c] for r in range(R)) for c in range(C)]
    tile = [sum(col[c] for c in range(64 * t, min(64 * t + 64, C))) for t in range(T)]
    row_bm = np.zeros((R, W64), dtype=np.uint64)
    for r in range(R):
        for t in range(T):
            if any(nz[r][c] for c in range(64 * t, min(64 * t + 64, C))):
                row_bm[r, t // 64] |= np.uint64(1) << np.uint64(t % 64)
    blk = np.zeros((RB, C32), dtype=np.uint32)
    for b in range(RB):
        for c in range(C):
            if any(nz[r][c] for r in range(128 * b, min(128 * b + 128, R))):
                blk[b, c // 32] |= np.uint32(1) << np.uint32(c % 32)
    return nnz, col, tile, row_bm, blk


@pytest.mark.parametrize("R,C,zp", [(1, 1, 0.5), (5, 7, 0.5), (130, 70, 0.7), (129, 65, 0.3),
                                    (3, 200, 0.5), (257, 33, 0.95), (2, 4200, 0.5)])
def test_stats_bruteforce(R, C, zp):
    rng = np.random.default_rng(R * 1000 + C)
    bits = _rand_bits((R, C), rng, zero_p=zp)
    st = orc.stats(bits, R, C)
    nnz, col, tile, row_bm, blk = _brute_stats(bits, R, C)
    assert st.nnz == nnz
    assert list(st.col_nnz) == col
    assert list(st.tile_nnz) == tile
    assert np.array_equal(st.row_bm, row_bm)
    assert np.array_equal(st.blk_mask, blk)
    assert st.sparsity == pytest.approx(1.0 - nnz / (R * C), abs=0)


def test_stats_special_cases():
    z = np.zeros((300, 100), dtype=np.uint16)
    z[::2, ::3] = 0x8000          # negative zeros are zeros
    st = orc.stats(z, 300, 100)
    assert st.nnz == 0 and st.sparsity == 1.0
    assert not st.row_bm.any() and not st.blk_mask.any()
    full = np.full((300, 100), 0x0001, dtype=np.uint16)   # smallest subnormal is non-zero
    st = orc.stats(full, 300, 100)
    assert st.nnz == 30000 and st.sparsity == 0.0
    assert all(st.col_nnz == 300)
    # padding bits past C and past R stay clear
    assert int(st.row_bm[0, 0]) == 0b11            # tiles 0 and 1 only (C = 100)
    assert int(st.blk_mask[2, 3]) == 0xF           # columns 96..99 only
    assert st.blk_mask.shape == (3, 4)


# ---------------------------------------------------------------------------
# Eq. 2 work: closed forms
# ---------------------------------------------------------------------------
def test_conv_work_closed_form():
    wk = orc.conv_work(8, 56, 56, 64, 64, 3, 3, 1, 1)
    assert (wk.Ho, wk.Wo) == (56, 56)
    assert wk.flops == 2 * 8 * 56 * 56 * 64 * 64 * 9 == 1_849_688_064
    assert wk.input_bytes == 8 * 56 * 56 * 64 * 2 == 3_211_264
    assert wk.flops_per_byte == 576.0
    assert wk.macs_eq2 == 3 * 3 * 64 * 64 * 56 * 56
    # stride 2, 7x7 stem of ResNet-18
    wk = orc.conv_work(1, 224, 224, 3, 64, 7, 7, 2, 3)
    assert (wk.Ho, wk.Wo) == (112, 112)
    assert wk.flops == 2 * 112 * 112 * 64 * 3 * 49
    # depthwise: FLOPs use C_in / groups, Eq. 2 uses C_in * C_out literally
    wk = orc.conv_work(2, 14, 14, 96, 96, 3, 3, 2, 1, groups=96)
    assert (wk.Ho, wk.Wo) == (7, 7)
    assert wk.flops == 2 * 2 * 7 * 7 * 96 * 1 * 9
    assert wk.macs_eq2 == 9 * 96 * 96 * 7 * 7


def test_fc_work_closed_form():
    wk = orc.fc_work(64, 512, 512)
    assert wk.flops == 33_554_432 and wk.input_bytes == 65_536 and wk.flops_per_byte == 512.0
    assert wk.macs_eq2 == 512 * 512


def _graph_flops(ops, x_shape):
    shapes = {0: x_shape}
    total = 0
    for i, op in enumerate(ops):
        s = shapes[op["input"]]
        if op["kind"] == "conv":
            N, H, W, C = s
            wk = orc.conv_work(N, H, W, C, op["cout"], op["k"], op["k"], op["stride"], op["pad"],
                               op["groups"])
            total += wk.flops
            shapes[i + 1] = (N, wk.Ho, wk.Wo, op["cout"])
        elif op["kind"] == "maxpool":
            N, H, W, C = s
            shapes[i + 1] = (N, (H + 2 * op["pad"] - op["k"]) // op["stride"] + 1,
                             (W + 2 * op["pad"] - op["k"]) // op["stride"] + 1, C)
        elif op["kind"] == "avgpool":
            shapes[i + 1] = (s[0], s[3])
        elif op["kind"] == "fc":
            total += orc.fc_work(s[0], s[1], op["cout"]).flops
            shapes[i + 1] = (s[0], op["cout"])
    return total


def test_resnet18_flops_match_table2():
    g = _golden("resnet18_table2.txt")
    ops, _, shape = synth.resnet18(batch=1)
    flops = _graph_flops(ops, shape)
    assert flops == 3_628_146_688          # closed form of the standard architecture
    gmacs = flops / 2 / 1e9
    assert round(gmacs, 1) == float(g["table2_gmacs"])   # Table 2: 1.8 G
    assert len(ops) == 23
    assert sum(op["kind"] == "conv" for op in ops) == 20


def test_mobilenet_v2_flops_closed_form():
    ops, _, shape = synth.mobilenet_v2(batch=1)
    flops = _graph_flops(ops, shape)
    # 300.8 M multiply-adds for MobileNetV2 1.0 at 224 (conv + FC)
    assert flops == 601_548_544
    assert sum(op["kind"] == "conv" for op in ops) == 52
    assert sum(op["kind"] == "conv" and op["groups"] > 1 for op in ops) == 17


# ---------------------------------------------------------------------------
# Threshold rule
# ---------------------------------------------------------------------------
def test_decide_thresholds_and_ties():
    # 1000 elements; s_thr 0.5 -> zero-skip iff zeros >= 500
    assert orc.decide(1000, 501, 100.0, 0, 0.5, 32.0) == orc.PATH_DENSE     # 499 zeros
    assert orc.decide(1000, 500, 100.0, 0, 0.5, 32.0) == orc.PATH_SKIP      # tie -> skip
    assert orc.decide(1000, 499, 100.0, 0, 0.5, 32.0) == orc.PATH_SKIP
    # below the sparsity threshold, intensity decides; tie -> dense
    assert orc.decide(1000, 900, 32.0, 0, 0.5, 32.0) == orc.PATH_DENSE
    assert orc.decide(1000, 900, math.nextafter(32.0, 0), 0, 0.5, 32.0) == orc.PATH_SKIP
    # forcing
    assert orc.decide(1000, 0, 1e9, 0, 0.5, 32.0, force_path=1) == orc.PATH_DENSE
    assert orc.decide(1000, 1000, 1e9, 0, 0.5, 32.0, force_path=2) == orc.PATH_SKIP
    # empty tensor: 0 zeros >= 0 -> skip
    assert orc.decide(0, 0, 0.0, 0, 0.5, 32.0) == orc.PATH_SKIP
    # s_thr 0 skips everything, s_thr > 1 never skips on sparsity
    assert orc.decide(10, 10, 1.0, 0, 0.0, 32.0) == orc.PATH_SKIP
    assert orc.decide(10, 0, 1e3, 0, 1.01, 32.0) == orc.PATH_DENSE


def test_decide_paper_quadrants_eq2_mode():
    q = _golden("quadrants.txt")
    ex = _golden("mdp_example.txt")
    s_thr, c_thr = float(q["s_thr"]), float(q["c_thr_eq2"])
    n = 10_000
    # Sec. 4.1 example: rho 0.2, I 1.8e11 -> dense (low sparsity, high intensity)
    nnz = int(round(n * (1 - float(ex["rho"]))))
    assert orc.decide(n, nnz, 0.0, int(float(ex["intensity"])), s_thr, c_thr, intensity_mode=1) == 1
    # BatchNorm-like: dense but light -> not the dense tensor-core path
    assert orc.decide(n, n, 0.0, 10 ** 6, s_thr, c_thr, intensity_mode=1) == 2
    # sparse (> 0.4) -> zero-skip even when heavy
    assert orc.decide(n, 5000, 0.0, 10 ** 9, s_thr, c_thr, intensity_mode=1) == 2


# ---------------------------------------------------------------------------
# Operators against library routines
# ---------------------------------------------------------------------------
def _t64(bits, shape):
    return torch.from_numpy(orc.bf16_to_f64(bits).reshape(shape))


def _torch_epilogue(y, bias, bn, eps, res, act):
    # y: [..., C] float64
    if bias is not None:
        y = y + torch.from_numpy(bias.astype(np.float64))
    if bn is not None:
        b = torch.from_numpy(bn.astype(np.float64))
        y = (y - b[2]) / torch.sqrt(b[3] + eps) * b[0] + b[1]
    if res is not None:
        y = y + res
    if act == 1:
        y = torch.clamp(y, min=0.0)
    elif act == 2:
        y = torch.clamp(y, 0.0, 6.0)
    return y


@pytest.mark.parametrize("N,H,W,Cin,Cout,k,stride,pad,groups,act,use_res", [
    (2, 9, 7, 8, 16, 3, 1, 1, 1, 1, True),
    (1, 11, 11, 3, 8, 7, 2, 3, 1, 1, False),
    (2, 8, 8, 16, 24, 1, 2, 0, 1, 0, False),
    (1, 10, 9, 12, 12, 3, 2, 1, 12, 2, False),     # depthwise, stride 2
    (3, 6, 6, 8, 8, 3, 1, 1, 8, 2, True),          # depthwise, residual
    (1, 5, 5, 6, 4, 3, 1, 0, 2, 0, False),         # grouped, no padding
])
def test_conv2d_vs_torch_float64(N, H, W, Cin, Cout, k, stride, pad, groups, act, use_res):
    rng = np.random.default_rng(N * 7 + H + Cin)
    g = torch.Generator().manual_seed(3)
    x = _rand_bits((N, H, W, Cin), rng, zero_p=0.4, specials=False)
    w = _rand_bits((Cout, k, k, Cin // groups), rng, zero_p=0.0, specials=False)
    bias = rng.standard_normal(Cout).astype(np.float32)
    bn = synth.random_bn(Cout, g)
    Ho = (H + 2 * pad - k) // stride + 1
    Wo = (W + 2 * pad - k) // stride + 1
    res = _rand_bits((N, Ho, Wo, Cout), rng, zero_p=0.2, specials=False) if use_res else None
    got = orc.conv2d(x, N, H, W, Cin, w, Cout, k, k, stride, pad, groups, bias, bn, 1e-5, res, act)
    xt = _t64(x, (N, H, W, Cin)).permute(0, 3, 1, 2)
    wt = _t64(w, (Cout, k, k, Cin // groups)).permute(0, 3, 1, 2)
    ref = F.conv2d(xt, wt, stride=stride, padding=pad, groups=groups).permute(0, 2, 3, 1)
    ref = _torch_epilogue(ref, bias, bn, 1e-5, _t64(res, (N, Ho, Wo, Cout)) if use_res else None, act)
    assert got.shape == tuple(ref.shape)
    np.testing.assert_allclose(got, ref.numpy(), rtol=1e-12, atol=1e-12)


def test_conv2d_vs_independent_im2col():
    rng = np.random.default_rng(11)
    N, H, W, Cin, Cout, k, s, p = 2, 7, 6, 5, 3, 3, 2, 1
    x = _rand_bits((N, H, W, Cin), rng, zero_p=0.3, specials=False)
    w = _rand_bits((Cout, k, k, Cin), rng, zero_p=0.0, specials=False)
    got = orc.conv2d(x, N, H, W, Cin, w, Cout, k, k, s, p)
    xv = orc.bf16_to_f64(x).reshape(N, H, W, Cin)
    xp = np.zeros((N, H + 2 * p, W + 2 * p, Cin))
    xp[:, p:p + H, p:p + W] = xv
    Ho, Wo = (H + 2 * p - k) // s + 1, (W + 2 * p - k) // s + 1
    cols = np.zeros((N, Ho, Wo, k, k, Cin))
    for i in range(Ho):
        for j in range(Wo):
            cols[:, i, j] = xp[:, i * s:i * s + k, j * s:j * s + k, :]
    ref = cols.reshape(N * Ho * Wo, -1) @ orc.bf16_to_f64(w).reshape(Cout, -1).T
    np.testing.assert_allclose(got.reshape(-1, Cout), ref, rtol=1e-12, atol=1e-12)


def test_fc_vs_numpy():
    rng = np.random.default_rng(5)
    M, K, N = 37, 70, 29
    x = _rand_bits((M, K), rng, zero_p=0.5, specials=False)
    w = _rand_bits((N, K), rng, zero_p=0.0, specials=False)
    bias = rng.standard_normal(N).astype(np.float32)
    res = _rand_bits((M, N), rng, zero_p=0.0, specials=False)
    got = orc.fc(x, M, K, w, N, bias=bias, residual_bits=res, act=1)
    ref = orc.bf16_to_f64(x).reshape(M, K) @ orc.bf16_to_f64(w).reshape(N, K).T
    ref = np.maximum(ref + bias.astype(np.float64) + orc.bf16_to_f64(res).reshape(M, N), 0.0)
    np.testing.assert_allclose(got, ref, rtol=1e-12, atol=1e-12)


def test_zero_skip_equals_dense_exactly():
    rng = np.random.default_rng(7)
    x = _rand_bits((2, 9, 9, 16), rng, zero_p=0.7, specials=False)
    w = _rand_bits((8, 3, 3, 16), rng, zero_p=0.0, specials=False)
    a = orc.conv2d(x, 2, 9, 9, 16, w, 8, 3, 3, 1, 1, skip_zeros=False)
    b = orc.conv2d(x, 2, 9, 9, 16, w, 8, 3, 3, 1, 1, skip_zeros=True)
    assert np.array_equal(a, b)
    xf = _rand_bits((33, 100), rng, zero_p=0.8, specials=False)
    wf = _rand_bits((20, 100), rng, zero_p=0.0, specials=False)
    assert np.array_equal(orc.fc(xf, 33, 100, wf, 20), orc.fc(xf, 33, 100, wf, 20, skip_zeros=True))


def test_maxpool_and_avgpool_vs_torch():
    rng = np.random.default_rng(9)
    x = _rand_bits((2, 13, 12, 8), rng, zero_p=0.3, specials=False)
    got = orc.maxpool(x, 2, 13, 12, 8, 3, 2, 1)
    xt = _t64(x, (2, 13, 12, 8)).permute(0, 3, 1, 2)
    ref = F.max_pool2d(xt, 3, 2, 1).permute(0, 2, 3, 1)
    assert np.array_equal(got, ref.numpy())
    got = orc.avgpool_global(x, 2, 13, 12, 8)
    ref = xt.mean(dim=(2, 3))
    np.testing.assert_allclose(got, ref.numpy(), rtol=1e-13)


def test_bn_act_vs_torch():
    rng = np.random.default_rng(10)
    g = torch.Generator().manual_seed(1)
    x = _rand_bits((50, 24), rng, zero_p=0.2, specials=False)
    bn = synth.random_bn(24, g)
    got = orc.bn_act(x, 50, 24, bn=bn, act=2)
    ref = _torch_epilogue(_t64(x, (50, 24)), None, bn, 1e-5, None, 2)
    np.testing.assert_allclose(got, ref.numpy(), rtol=1e-12, atol=1e-12)


def test_run_graph_composes_ops():
    """A two-op graph equals the ops applied by hand with bf16 rounding between."""
    g = torch.Generator().manual_seed(4)
    rng = np.random.default_rng(4)
    x = _rand_bits((1, 8, 8, 8), rng, zero_p=0.5, specials=False)
    op1 = synth._conv_op(g, 0, 8, 16, 3, 1, 1, synth.ACT_RELU)
    op2 = synth._conv_op(g, 1, 16, 8, 1, 1, 0, synth.ACT_NONE, residual=0)
    recs = orc.run_graph([op1, op2], x, (1, 8, 8, 8))
    y1 = orc.f64_to_bf16(orc.conv2d(x, 1, 8, 8, 8, op1["w"], 16, 3, 3, 1, 1, bn=op1["bn"], act=1))
    y2 = orc.conv2d(y1, 1, 8, 8, 16, op2["w"], 8, 1, 1, 1, 0, bn=op2["bn"], residual_bits=x)
    assert np.array_equal(recs[0].out_bits, y1)
    assert np.array_equal(recs[1].out_f64, y2)
    assert recs[0].in_stats.nnz == orc.stats(x, 64, 8).nnz
