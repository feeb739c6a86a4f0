"""Split execution of an FC operator (zero-skip rows + dense rows on two
streams) against the oracle, and its output occupancy assembled from both parts."""
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


def _case(M, K, N, seed):
    g = torch.Generator().manual_seed(seed)
    # block-structured zeros in the first half of the rows, dense second half
    h = synth.structured_activation((M, K), 0.8, "block", g).float()
    h[M // 2:] = torch.randn(M - M // 2, K, generator=g).abs() + 1e-3
    xb = synth.to_bf16_bits(h)
    wb = synth.to_bf16_bits(torch.randn(N, K, generator=g) / np.sqrt(K))
    bias = (0.1 * torch.randn(N, generator=g)).numpy().astype(np.float32)
    bn = synth.random_bn(N, g)
    return xb, wb, bias, bn


@pytest.mark.parametrize("M,K,N", [(300, 512, 256), (64, 512, 512), (1024, 3072, 768)])
@pytest.mark.parametrize("xi", [0.0, 0.3, 0.5, 1.0])
def test_split_matches_oracle(sp, ctx, M, K, N, xi):
    xb, wb, bias, bn = _case(M, K, N, M + K + N)
    x = sp.bits_to_device(xb).view(M, K)
    W = sp.bits_to_device(wb).view(N, K)
    W_kn = W.t().contiguous()
    y = torch.empty(M, N, dtype=torch.bfloat16, device="cuda")
    yo = sp.OccupancyBuffer(M, N)
    sp.sparoa_gemm_split(ctx, x, W, y, xi, W_kn=W_kn, bias=torch.from_numpy(bias).cuda(),
                         bn=torch.from_numpy(bn).cuda(), act=sp.ACT_RELU, y_occ=yo)
    torch.cuda.synchronize()
    ybits = sp.device_to_bits(y)
    rows = np.arange(M) if M <= 300 else np.sort(np.random.default_rng(0).choice(M, 96, replace=False))
    ref = orc.fc(xb.reshape(M, K)[rows], len(rows), K, wb, N, bias=bias, bn=bn, act=1)
    got = synth.bits_to_f32(ybits).astype(np.float64).reshape(M, N)[rows]
    assert_close(got, ref, what=f"split {M}x{K}x{N} xi={xi}")
    assert_occ_equal(yo.to_host(), orc.stats(ybits, M, N), f"split y_occ xi={xi}")


def test_split_equals_unsplit_dense_and_skip(sp, ctx):
    M, K, N = 512, 1024, 256
    xb, wb, bias, bn = _case(M, K, N, 7)
    x = sp.bits_to_device(xb).view(M, K)
    W = sp.bits_to_device(wb).view(N, K)
    ys = {}
    for tag, call in (("dense", lambda y: sp.sparoa_gemm(ctx, x, W, y, thr=sp.thresholds(force_path=1))),
                      ("skip", lambda y: sp.sparoa_gemm(ctx, x, W, y, thr=sp.thresholds(force_path=2))),
                      ("split", lambda y: sp.sparoa_gemm_split(ctx, x, W, y, 0.5))):
        y = torch.empty(M, N, dtype=torch.bfloat16, device="cuda")
        call(y)
        ys[tag] = y.float().cpu().numpy()
    # the two tensor-core paths sum in the same order (skipped blocks only add
    # zeros), so they agree exactly; the split's halves may pick another K
    # split for their smaller M, so it agrees to bf16 rounding
    assert np.array_equal(ys["dense"], ys["skip"])
    scale = np.abs(ys["dense"]).max()
    assert np.abs(ys["split"] - ys["dense"]).max() <= 1e-2 * scale


def test_split_under_graph_capture(sp, ctx):
    M, K, N = 512, 512, 128
    xb, wb, _, _ = _case(M, K, N, 11)
    x = sp.bits_to_device(xb).view(M, K)
    W = sp.bits_to_device(wb).view(N, K)
    y = torch.empty(M, N, dtype=torch.bfloat16, device="cuda")
    xo = sp.OccupancyBuffer(M, K)
    sp.sparoa_op_stats(ctx, x, (M, K), occ=xo, host=False)
    sp.sparoa_gemm_split(ctx, x, W, y, 0.5, x_occ=xo)
    torch.cuda.synchronize()
    want = y.clone()
    y.zero_()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g):
        sp.sparoa_gemm_split(ctx, x, W, y, 0.5, x_occ=xo)
    g.replay()
    torch.cuda.synchronize()
    assert torch.equal(y, want)


def test_split_rejects_bad_fraction(sp, ctx):
    x = torch.zeros(128, 64, dtype=torch.bfloat16, device="cuda")
    W = torch.zeros(64, 64, dtype=torch.bfloat16, device="cuda")
    y = torch.empty(128, 64, dtype=torch.bfloat16, device="cuda")
    with pytest.raises(sp.SparoaError):
        sp.sparoa_gemm_split(ctx, x, W, y, 1.5)
