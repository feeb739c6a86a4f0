"""Parity of every libsparoa operator with the oracle, through the C ABI (GPU).

Integers (Eq. 1 counts, bitmaps, dispatch decisions, max pooling) must match
bit for bit; floats within max|err| <= 2e-2*max|ref| and relative Frobenius
error <= 5e-3 (bf16 inputs, fp32 accumulation).  Output occupancy written by
the fused epilogues is compared with the oracle's statistics of the very bf16
tensor the GPU produced.
"""
import numpy as np
import pytest
import torch

from oracle import oracle as orc
from paper_2511_19457_gb300 import synth
from tests._parity import assert_close, assert_occ_equal

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def sp():
    from paper_2511_19457_gb300 import sparoa
    return sparoa


@pytest.fixture(scope="module")
def ctx(sp):
    c = sp.Context(0)
    yield c
    c.close()


def _bits(shape, seed, zero_p=0.5, dist="normal"):
    g = torch.Generator().manual_seed(seed)
    v = torch.randn(*shape, generator=g)
    if dist == "abs":
        v = v.abs()
    z = torch.rand(*shape, generator=g) < zero_p
    v[z] = 0.0
    return synth.to_bf16_bits(v)


def _dev(sp, bits, shape):
    return sp.bits_to_device(bits).view(*shape)


def _f64(t):
    return t.float().cpu().numpy().astype(np.float64)


# ---------------------------------------------------------------------------
# Eq. 1 statistics
# ---------------------------------------------------------------------------
@pytest.mark.parametrize("R,C,zp", [(1, 8, 0.5), (64, 512, 0.7), (130, 72, 0.5), (257, 40, 0.9),
                                    (129, 70, 0.5), (50176, 3, 0.1), (25088, 64, 0.5),
                                    (300, 4104, 0.3), (200, 64, 0.0), (200, 64, 1.0),
                                    # narrow tensors (C < 8): whole and partial 8-row groups,
                                    # blocks split between half warps, many blocks
                                    (1, 3, 0.5), (7, 3, 0.5), (1001, 1, 0.5), (999, 2, 0.3),
                                    (50177, 3, 0.5), (4097, 5, 0.7), (131, 6, 0.2), (12345, 7, 0.9),
                                    (1605632, 3, 0.0)])
def test_stats_bit_exact(sp, ctx, R, C, zp):
    bits = _bits((R, C), R + C, zero_p=zp)
    if R * C > 16:
        flat = bits.reshape(-1)
        flat[:5] = [0x8000, 0x0001, 0x7FC0, 0xFF80, 0x8001]   # -0, subnormals, NaN, -inf
    x = _dev(sp, bits, (R, C))
    occ = sp.OccupancyBuffer(R, C)
    st = sp.sparoa_op_stats(ctx, x, (R, C), occ=occ, host=True)
    ref = orc.stats(bits, R, C)
    assert st.nnz == ref.nnz and st.numel == R * C
    assert st.sparsity == pytest.approx(ref.sparsity, abs=0)
    assert_occ_equal(occ.to_host(), ref, f"stats {R}x{C}")


def test_stats_needs_no_cleared_output_and_repeats(sp, ctx):
    """The stats kernel writes every occupancy field (a buffer full of junk
    comes out exact), and back-to-back launches on one context agree with the
    oracle each time (its column accumulator is left clean), including more
    row blocks than CTAs."""
    for (R, C, zp, seed) in [(100352, 64, 0.5, 1), (100352, 64, 0.8, 2), (777, 136, 0.3, 3),
                             (300, 4104, 0.6, 4)]:
        bits = _bits((R, C), seed, zero_p=zp)
        x = _dev(sp, bits, (R, C))
        occ = sp.OccupancyBuffer(R, C)
        occ.buf.fill_(0xA5)
        st = sp.sparoa_op_stats(ctx, x, (R, C), occ=occ, host=True)
        ref = orc.stats(bits, R, C)
        assert st.nnz == ref.nnz
        assert_occ_equal(occ.to_host(), ref, f"stats junk-filled {R}x{C}")


def test_stats_reports_consumer_work(sp, ctx):
    d = synth.conv_layer(seed=0)
    x = _dev(sp, d["x"], (8, 56, 56, 64))
    op = sp.Op(kind=sp.OP_CONV2D, c_in=64, c_out=64, kh=3, kw=3, stride=1, pad=1, groups=1,
               thr=sp.thresholds())
    st = sp.sparoa_op_stats(ctx, x, (8, 56, 56, 64), consumer=op)
    wk = orc.conv_work(8, 56, 56, 64, 64, 3, 3, 1, 1)
    ref = orc.stats(d["x"], 8 * 56 * 56, 64)
    assert (st.flops, st.macs_eq2, st.input_bytes) == (wk.flops, wk.macs_eq2, wk.input_bytes)
    assert st.flops_per_byte == wk.flops_per_byte == 576.0
    assert st.path == orc.decide(ref.numel, ref.nnz, wk.flops_per_byte, wk.macs_eq2, 0.5, 32.0)
    assert (st.B, st.C_in, st.H, st.W) == (8, 64, 56, 56)


# ---------------------------------------------------------------------------
# fully connected
# ---------------------------------------------------------------------------
@pytest.mark.parametrize("force,with_kn", [(0, True), (1, True), (2, True), (2, False)])
def test_fc_layer_fp32(sp, ctx, force, with_kn):
    d = synth.fc_layer(seed=0)
    x = _dev(sp, d["x"], (64, 512))
    w = _dev(sp, d["w"], (512, 512))
    wkn = _dev(sp, d["w_kn"], (512, 512)) if with_kn else None
    bias = torch.from_numpy(d["bias"]).cuda()
    y = torch.empty(64, 512, dtype=torch.float32, device="cuda")
    st = sp.sparoa_gemm(ctx, x, w, y, W_kn=wkn, bias=bias, thr=sp.thresholds(force_path=force),
                        host=True)
    ref_st = orc.stats(d["x"], 64, 512)
    wk = orc.fc_work(64, 512, 512)
    assert st.nnz == ref_st.nnz
    assert st.path == orc.decide(ref_st.numel, ref_st.nnz, wk.flops_per_byte, wk.macs_eq2, 0.5, 32.0,
                                 0, force)
    if force == 0:
        assert st.path == sp.PATH_SKIP          # about 70% zeros >= 0.5
    ref = orc.fc(d["x"], 64, 512, d["w"], 512, bias=d["bias"])
    assert_close(_f64(y), ref, what=f"fc force={force}")


@pytest.mark.parametrize("M,K,N", [(200, 136, 72), (1, 512, 1000), (128, 64, 64), (300, 1280, 200),
                                   (260, 4096, 136), (256, 3072, 768),  # few tiles, split K
                                   (4096, 256, 712),   # 192-wide tiles, ragged last column tile
                                   (6304, 128, 768)])  # 256-wide tiles, ragged last row tile
@pytest.mark.parametrize("force", [1, 2])
def test_gemm_epilogue_and_occupancy(sp, ctx, M, K, N, force):
    g = torch.Generator().manual_seed(M + K + N)
    xb = _bits((M, K), M * 7 + K, zero_p=0.6, dist="abs")
    wb = synth.to_bf16_bits(torch.randn(N, K, generator=g) / np.sqrt(K))
    wkn = synth.to_bf16_bits(torch.from_numpy(synth.bits_to_f32(wb)).t().contiguous())
    bias = (0.1 * torch.randn(N, generator=g)).numpy().astype(np.float32)
    bn = synth.random_bn(N, g)
    resb = _bits((M, N), M + 3, zero_p=0.3)
    x = _dev(sp, xb, (M, K))
    y = torch.empty(M, N, dtype=torch.bfloat16, device="cuda")
    yo = sp.OccupancyBuffer(M, N)
    st = sp.sparoa_gemm(ctx, x, _dev(sp, wb, (N, K)), y, W_kn=_dev(sp, wkn, (K, N)),
                        bias=torch.from_numpy(bias).cuda(), bn=torch.from_numpy(bn).cuda(),
                        act=sp.ACT_RELU, residual=_dev(sp, resb, (M, N)),
                        thr=sp.thresholds(force_path=force), y_occ=yo, host=True)
    assert st.path == force
    ref = orc.fc(xb, M, K, wb, N, bias=bias, bn=bn, residual_bits=resb, act=1)
    assert_close(_f64(y), ref, what=f"gemm {M}x{K}x{N} force={force}")
    ybits = sp.device_to_bits(y)
    assert_occ_equal(yo.to_host(), orc.stats(ybits, M, N), "gemm y_occ")


@pytest.mark.parametrize("structure", ["block32", "unstructured"])
@pytest.mark.parametrize("force", [1, 2])
def test_mlp_down_projection(sp, ctx, structure, force):
    """768 <- 3072 down projection at 50% activation sparsity, M = 1024 tokens;
    checked on a seeded sample of 64 rows (the fp64 oracle on all rows is slow)."""
    M = 1024
    wts = synth.mlp_weights(seed=0)
    hb = synth.mlp_hidden(M, 0.5, structure, seed=1)
    h = _dev(sp, hb, (M, 3072))
    y = torch.empty(M, 768, dtype=torch.bfloat16, device="cuda")
    st = sp.sparoa_gemm(ctx, h, _dev(sp, wts["w2"], (768, 3072)), y,
                        thr=sp.thresholds(force_path=force), host=True)
    assert st.path == force
    rows = np.sort(np.random.default_rng(0).choice(M, 64, replace=False))
    sub = hb.reshape(M, 3072)[rows]
    ref = orc.fc(sub, 64, 3072, wts["w2"], 768)
    assert_close(_f64(y)[rows], ref, what=f"mlp {structure} force={force}")


def test_gemm_all_zero_input_skip_path(sp, ctx):
    M, K, N = 256, 512, 128
    x = torch.zeros(M, K, dtype=torch.bfloat16, device="cuda")
    w = torch.randn(N, K, device="cuda").to(torch.bfloat16)
    bias = torch.linspace(-1, 1, N, device="cuda")
    y = torch.empty(M, N, dtype=torch.float32, device="cuda")
    st = sp.sparoa_gemm(ctx, x, w, y, bias=bias, host=True)
    assert st.nnz == 0 and st.path == sp.PATH_SKIP
    assert torch.equal(y, bias.expand(M, N))


def test_gemm_empty_batch(sp, ctx):
    x = torch.empty(0, 64, dtype=torch.bfloat16, device="cuda")
    w = torch.randn(64, 64, device="cuda").to(torch.bfloat16)
    y = torch.empty(0, 64, dtype=torch.bfloat16, device="cuda")
    st = sp.sparoa_gemm(ctx, x, w, y, host=True)
    assert st.numel == 0 and st.nnz == 0


# ---------------------------------------------------------------------------
# convolution
# ---------------------------------------------------------------------------
@pytest.mark.parametrize("force", [0, 1, 2])
def test_conv_layer(sp, ctx, force):
    d = synth.conv_layer(seed=0)
    x = _dev(sp, d["x"], (8, 56, 56, 64))
    w = _dev(sp, d["w"], (64, 3, 3, 64))
    y = torch.empty(8, 56, 56, 64, dtype=torch.bfloat16, device="cuda")
    yo = sp.OccupancyBuffer(8 * 56 * 56, 64)
    st = sp.sparoa_conv2d(ctx, x, w, y, stride=1, pad=1, bn=torch.from_numpy(d["bn"]).cuda(),
                          act=sp.ACT_RELU, thr=sp.thresholds(force_path=force), y_occ=yo, host=True)
    ref_st = orc.stats(d["x"], 8 * 56 * 56, 64)
    wk = orc.conv_work(8, 56, 56, 64, 64, 3, 3, 1, 1)
    assert st.nnz == ref_st.nnz
    assert st.path == orc.decide(ref_st.numel, ref_st.nnz, wk.flops_per_byte, wk.macs_eq2, 0.5, 32.0,
                                 0, force)
    ref = orc.conv2d(d["x"], 8, 56, 56, 64, d["w"], 64, 3, 3, 1, 1, bn=d["bn"], act=1)
    assert_close(_f64(y), ref, what=f"conv force={force}")
    assert_occ_equal(yo.to_host(), orc.stats(sp.device_to_bits(y), 8 * 56 * 56, 64), "conv y_occ")


CONV_CASES = [
    # N, H, W, Cin, Cout, k, stride, pad, act, residual
    (2, 15, 17, 64, 128, 3, 2, 1, 1, False),
    (2, 14, 14, 96, 24, 1, 1, 0, 0, True),     # pointwise (TMA GEMM mode), linear + residual
    (2, 9, 10, 64, 40, 1, 1, 0, 2, True),      # residual over a block of 8 of 32 columns
    (2, 14, 14, 64, 128, 1, 2, 0, 0, False),   # strided 1x1 downsample
    (1, 32, 30, 3, 64, 7, 2, 3, 1, False),     # stem, C_in padded to 8
    (3, 21, 19, 3, 32, 3, 2, 1, 2, False),     # 3x3 stem; 1197 pixels: a partial 8-pixel group
    (2, 9, 13, 5, 16, 3, 1, 1, 0, False),      # C_in 5
    (2, 9, 11, 144, 32, 1, 1, 0, 2, False),    # K = 144 (ragged 32-block)
    (2, 10, 10, 24, 144, 3, 1, 1, 2, False),   # C_in 24: blocks straddle taps
    (1, 7, 7, 512, 512, 3, 1, 1, 1, True),
    # spatial output tiles whose 32-row epilogue blocks are {4 w, 4 h, 2 images},
    # {32 of 128 w}, and several whole images
    (8, 6, 6, 64, 64, 3, 2, 1, 1, False),
    (1, 8, 128, 64, 128, 3, 1, 1, 1, True),
    (32, 8, 8, 64, 64, 3, 2, 1, 0, False),
]


@pytest.mark.parametrize("case", CONV_CASES)
@pytest.mark.parametrize("force", [1, 2])
def test_conv_shapes(sp, ctx, case, force):
    N, H, W, Cin, Cout, k, s, p, act, use_res = case
    g = torch.Generator().manual_seed(N * H + Cin + Cout)
    xb = _bits((N, H, W, Cin), H * W + Cin, zero_p=0.5, dist="abs")
    wb = synth.to_bf16_bits(synth.he_normal((Cout, k, k, Cin), Cin * k * k, g))
    bn = synth.random_bn(Cout, g)
    Ho, Wo = (H + 2 * p - k) // s + 1, (W + 2 * p - k) // s + 1
    resb = _bits((N, Ho, Wo, Cout), Cout, zero_p=0.2) if use_res else None
    y = torch.empty(N, Ho, Wo, Cout, dtype=torch.bfloat16, device="cuda")
    yo = sp.OccupancyBuffer(N * Ho * Wo, Cout)
    st = sp.sparoa_conv2d(ctx, _dev(sp, xb, (N, H, W, Cin)), _dev(sp, wb, (Cout, k, k, Cin)), y,
                          stride=s, pad=p, bn=torch.from_numpy(bn).cuda(), act=act,
                          residual=_dev(sp, resb, (N, Ho, Wo, Cout)) if use_res else None,
                          thr=sp.thresholds(force_path=force), y_occ=yo, host=True)
    assert st.path == force
    ref = orc.conv2d(xb, N, H, W, Cin, wb, Cout, k, k, s, p, bn=bn, residual_bits=resb, act=act)
    assert_close(_f64(y), ref, what=f"conv {case} force={force}")
    assert_occ_equal(yo.to_host(), orc.stats(sp.device_to_bits(y), N * Ho * Wo, Cout), "y_occ")


def test_conv_structured_zeros_skip_equals_dense(sp, ctx):
    """Whole 64-channel tiles of the input zero over large regions: the
    zero-skip path really leaves K blocks out, and still equals the oracle."""
    N, H, W, C = 2, 24, 24, 128
    g = torch.Generator().manual_seed(5)
    x = torch.randn(N, H, W, C, generator=g).abs()
    x[:, :, :, 64:] = 0.0          # second channel tile empty everywhere
    x[:, :12] = 0.0                # top half of every image empty
    xb = synth.to_bf16_bits(x)
    wb = synth.to_bf16_bits(synth.he_normal((64, 3, 3, C), 9 * C, g))
    outs = []
    for force in (1, 2):
        y = torch.empty(N, H, W, 64, dtype=torch.bfloat16, device="cuda")
        sp.sparoa_conv2d(ctx, _dev(sp, xb, (N, H, W, C)), _dev(sp, wb, (64, 3, 3, C)), y, stride=1,
                         pad=1, thr=sp.thresholds(force_path=force), host=True)
        outs.append(_f64(y))
    ref = orc.conv2d(xb, N, H, W, C, wb, 64, 3, 3, 1, 1)
    assert_close(outs[0], ref, what="dense")
    assert_close(outs[1], ref, what="skip")


# ---------------------------------------------------------------------------
# depthwise, pooling, batch norm
# ---------------------------------------------------------------------------
@pytest.mark.parametrize("N,H,W,C,s,act,res", [
    (2, 17, 15, 96, 1, 2, False), (2, 17, 15, 96, 2, 2, False), (1, 8, 8, 8, 1, 2, False),
    (3, 14, 14, 960, 1, 2, False),
    # every activation and a residual; C = 32 and 144 leave a partial 64-channel slice
    (4, 29, 31, 32, 2, 0, False), (2, 11, 9, 144, 1, 1, True), (2, 12, 20, 48, 2, 3, False),
    (1, 7, 7, 576, 2, 2, True),
    # enough pixel tiles that every CTA runs all slices of its tiles (owned row words)
    (32, 56, 56, 144, 1, 2, False), (32, 112, 112, 96, 2, 2, False)])
def test_depthwise(sp, ctx, N, H, W, C, s, act, res):
    g = torch.Generator().manual_seed(C + s)
    xb = _bits((N, H, W, C), C * s, zero_p=0.5, dist="abs")
    wb = synth.to_bf16_bits(synth.he_normal((C, 3, 3, 1), 9, g))
    bn = synth.random_bn(C, g)
    Ho, Wo = (H + 2 - 3) // s + 1, (W + 2 - 3) // s + 1
    rb = _bits((N, Ho, Wo, C), C + 7, zero_p=0.3) if res else None
    y = torch.empty(N, Ho, Wo, C, dtype=torch.bfloat16, device="cuda")
    yo = sp.OccupancyBuffer(N * Ho * Wo, C)
    st = sp.sparoa_conv2d(ctx, _dev(sp, xb, (N, H, W, C)), _dev(sp, wb, (C, 3, 3, 1)), y, stride=s,
                          pad=1, groups=C, bn=torch.from_numpy(bn).cuda(), act=act,
                          residual=_dev(sp, rb, (N, Ho, Wo, C)) if res else None, y_occ=yo, host=True)
    assert st.path == sp.PATH_DEPTHWISE
    assert st.nnz == orc.stats(xb, N * H * W, C).nnz
    ref = orc.conv2d(xb, N, H, W, C, wb, C, 3, 3, s, 1, groups=C, bn=bn, residual_bits=rb, act=act)
    assert_close(_f64(y), ref, what="depthwise")
    assert_occ_equal(yo.to_host(), orc.stats(sp.device_to_bits(y), N * Ho * Wo, C), "dw y_occ")


@pytest.mark.parametrize("shape", [(2, 33, 31, 64), (3, 9, 11, 128), (4, 112, 112, 64), (1, 2, 3, 8)])
def test_maxpool_bit_exact(sp, ctx, shape):
    """Interior windows (fixed tap offsets) and border windows (clamped taps),
    output rows that wrap several image rows per 32-row step (Wo = 5, 6),
    two column tiles, many tiles, and a window larger than the image."""
    N, H, W, C = shape
    xb = _bits((N, H, W, C), 9, zero_p=0.4)
    Ho, Wo = (H + 2 - 3) // 2 + 1, (W + 2 - 3) // 2 + 1
    y = torch.empty(N, Ho, Wo, C, dtype=torch.bfloat16, device="cuda")
    yo = sp.OccupancyBuffer(N * Ho * Wo, C)
    sp.sparoa_maxpool2d(ctx, _dev(sp, xb, (N, H, W, C)), y, 3, 2, 1, y_occ=yo)
    ref = orc.maxpool(xb, N, H, W, C, 3, 2, 1)
    got = _f64(y)
    assert np.array_equal(got.reshape(ref.shape), ref)
    assert_occ_equal(yo.to_host(), orc.stats(sp.device_to_bits(y), N * Ho * Wo, C), "maxpool y_occ")


def test_avgpool(sp, ctx):
    N, H, W, C = 5, 7, 7, 520
    xb = _bits((N, H, W, C), 10, zero_p=0.5, dist="abs")
    y = torch.empty(N, C, dtype=torch.bfloat16, device="cuda")
    yo = sp.OccupancyBuffer(N, C)
    sp.sparoa_avgpool_global(ctx, _dev(sp, xb, (N, H, W, C)), y, y_occ=yo)
    assert_close(_f64(y), orc.avgpool_global(xb, N, H, W, C), what="avgpool")
    assert_occ_equal(yo.to_host(), orc.stats(sp.device_to_bits(y), N, C), "avgpool y_occ")


@pytest.mark.parametrize("R,C", [(300, 72), (1000, 64)])
@pytest.mark.parametrize("with_res", [False, True])
@pytest.mark.parametrize("act", [0, 1, 2, 3])
def test_bn_act(sp, ctx, R, C, with_res, act):
    """Every activation, with and without a residual (the kernel's
    compile-time variants), on one and on two column tiles."""
    g = torch.Generator().manual_seed(2)
    xb = _bits((R, C), 11, zero_p=0.3)
    rb = _bits((R, C), 12, zero_p=0.3)
    bn = synth.random_bn(C, g)
    y = torch.empty(R, C, dtype=torch.bfloat16, device="cuda")
    yo = sp.OccupancyBuffer(R, C)
    sp.sparoa_bn_act(ctx, _dev(sp, xb, (R, C)), y, bn=torch.from_numpy(bn).cuda(), act=act,
                     residual=_dev(sp, rb, (R, C)) if with_res else None, y_occ=yo)
    ref = orc.bn_act(xb, R, C, bn=bn, residual_bits=rb if with_res else None, act=act)
    assert_close(_f64(y), ref, what=f"bn_act act {act} residual {with_res}")
    assert_occ_equal(yo.to_host(), orc.stats(sp.device_to_bits(y), R, C), "bn_act y_occ")


# ---------------------------------------------------------------------------
# argument errors come back as status codes
# ---------------------------------------------------------------------------
def test_invalid_arguments_return_status(sp, ctx):
    x = torch.zeros(64, 60, dtype=torch.bfloat16, device="cuda")   # K % 8 != 0
    w = torch.zeros(64, 60, dtype=torch.bfloat16, device="cuda")
    y = torch.empty(64, 64, dtype=torch.bfloat16, device="cuda")
    with pytest.raises(sp.SparoaError) as e:
        sp.sparoa_gemm(ctx, x, w, y)
    assert e.value.status == sp.ERR_INVALID_ARG
    xg = torch.zeros(1, 8, 8, 16, dtype=torch.bfloat16, device="cuda")
    wg = torch.zeros(16, 3, 3, 8, dtype=torch.bfloat16, device="cuda")
    yg = torch.empty(1, 8, 8, 16, dtype=torch.bfloat16, device="cuda")
    with pytest.raises(sp.SparoaError) as e:
        sp.sparoa_conv2d(ctx, xg, wg, yg, stride=1, pad=1, groups=2)
    assert e.value.status == sp.ERR_UNSUPPORTED
    with pytest.raises(sp.SparoaError) as e:
        sp.sparoa_gemm(ctx, torch.zeros(8, 64, dtype=torch.bfloat16, device="cuda"),
                       torch.zeros(64, 64, dtype=torch.bfloat16, device="cuda"),
                       torch.empty(8, 64, dtype=torch.bfloat16, device="cuda"),
                       thr=sp.thresholds(force_path=7))
    assert e.value.status == sp.ERR_INVALID_ARG
    ctx.sync()   # the context stays usable


# 3x3 stride-1 convolutions with resident weights and per-tile input slabs
CONV3_CASES = [
    # N, H, W, Cin, Cout, act, residual
    (1, 7, 9, 64, 64, 1, True),
    (2, 30, 17, 32, 128, 2, False),
    (1, 20, 112, 64, 64, 1, False),
    (3, 5, 5, 16, 64, 0, True),
    (8, 56, 56, 64, 64, 1, True),   # 208 tiles: several per persistent CTA
]


@pytest.mark.parametrize("case", CONV3_CASES)
@pytest.mark.parametrize("force", [1, 2])
def test_conv3x3_slab_kernel(sp, ctx, case, force):
    N, H, W, Cin, Cout, act, use_res = case
    g = torch.Generator().manual_seed(H * W + Cin + Cout)
    xb = _bits((N, H, W, Cin), H * 31 + W, zero_p=0.5, dist="abs")
    wb = synth.to_bf16_bits(synth.he_normal((Cout, 3, 3, Cin), Cin * 9, g))
    bn = synth.random_bn(Cout, g)
    bias = (0.1 * torch.randn(Cout, generator=g)).numpy().astype(np.float32)
    resb = _bits((N, H, W, Cout), Cout + 1, zero_p=0.2) if use_res else None
    y = torch.empty(N, H, W, Cout, dtype=torch.bfloat16, device="cuda")
    yo = sp.OccupancyBuffer(N * H * W, Cout)
    st = sp.sparoa_conv2d(ctx, _dev(sp, xb, (N, H, W, Cin)), _dev(sp, wb, (Cout, 3, 3, Cin)), y,
                          stride=1, pad=1, bias=torch.from_numpy(bias).cuda(),
                          bn=torch.from_numpy(bn).cuda(), act=act,
                          residual=_dev(sp, resb, (N, H, W, Cout)) if use_res else None,
                          thr=sp.thresholds(force_path=force), y_occ=yo, host=True)
    assert st.path == force
    ref = orc.conv2d(xb, N, H, W, Cin, wb, Cout, 3, 3, 1, 1, bias=bias, bn=bn, residual_bits=resb,
                     act=act)
    assert_close(_f64(y), ref, what=f"conv3 {case} force={force}")
    assert_occ_equal(yo.to_host(), orc.stats(sp.device_to_bits(y), N * H * W, Cout), "conv3 y_occ")


def test_conv3x3_slab_kernel_skips_zero_regions(sp, ctx):
    """Top half of every image and one whole image all zero: the zero-skip path
    leaves out those taps' MMAs and still matches the oracle (including tiles
    whose every tap is unoccupied)."""
    N, H, W, C = 3, 24, 24, 64
    g = torch.Generator().manual_seed(8)
    x = torch.randn(N, H, W, C, generator=g).abs()
    x[:, :12] = 0.0
    x[1] = 0.0
    xb = synth.to_bf16_bits(x)
    wb = synth.to_bf16_bits(synth.he_normal((64, 3, 3, C), 9 * C, g))
    outs = []
    for force in (1, 2):
        y = torch.empty(N, H, W, 64, dtype=torch.bfloat16, device="cuda")
        sp.sparoa_conv2d(ctx, _dev(sp, xb, (N, H, W, C)), _dev(sp, wb, (64, 3, 3, C)), y, stride=1,
                         pad=1, act=1, thr=sp.thresholds(force_path=force), host=True)
        outs.append(_f64(y))
    ref = orc.conv2d(xb, N, H, W, C, wb, 64, 3, 3, 1, 1, act=1)
    assert_close(outs[0], ref, what="dense")
    assert_close(outs[1], ref, what="skip")
