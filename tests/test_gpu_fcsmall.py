"""The fused small-FC path on the GPU: statistics, dispatch and the zero-skip
product in one kernel for inputs that fit shared memory whole (M <= 128).

Checked against the oracle: the Eq. 1 count (Sec. 3.1) the kernel measures
itself, the path of the Sec. 3 rule on that count, the output, and the output
occupancy, over row counts that leave k-step groups of every size (M = 1, 16,
48, 100, 128), K that is not a multiple of 16, N that is not a multiple of 16,
whole zero columns, an all-zero input, GELU, and with the input's occupancy
given by the caller instead of measured.
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


def _case(M, K, N, zero_p, col_p, seed):
    g = torch.Generator().manual_seed(seed)
    x = torch.relu(torch.randn(M, K, generator=g))
    x = x * (torch.rand(M, K, generator=g) >= zero_p).to(torch.float32)
    x = x * (torch.rand(K, generator=g) >= col_p).to(torch.float32)[None, :]
    w = torch.randn(N, K, generator=g) / np.sqrt(K)
    bias = (0.1 * torch.randn(N, generator=g)).numpy().astype(np.float32)
    return synth.to_bf16_bits(x), synth.to_bf16_bits(w), synth.to_bf16_bits(w.t().contiguous()), bias


@pytest.mark.parametrize("M,K,N", [(1, 520, 40), (16, 24, 8), (48, 1000, 72), (100, 512, 136),
                                   (128, 256, 64), (64, 512, 512)])
@pytest.mark.parametrize("force", [0, 1, 2])
@pytest.mark.parametrize("given_occ", [False, True])
def test_fused_small_fc(sp, ctx, M, K, N, force, given_occ):
    xb, wb, wknb, bias = _case(M, K, N, 0.3, 0.4, M * 13 + K + N)
    x = sp.bits_to_device(xb).view(M, K)
    y = torch.full((M, N), float("nan"), dtype=torch.bfloat16, device="cuda")
    yo = sp.OccupancyBuffer(M, N)
    xo = None
    if given_occ:
        xo = sp.OccupancyBuffer(M, K)
        sp.sparoa_op_stats(ctx, x, (M, K), occ=xo, host=False)
    st = sp.sparoa_gemm(ctx, x, sp.bits_to_device(wb).view(N, K), y, W_kn=sp.bits_to_device(wknb).view(K, N),
                        bias=torch.from_numpy(bias).cuda(), act=sp.ACT_GELU,
                        thr=sp.thresholds(force_path=force), x_occ=xo, y_occ=yo, host=True)
    ref_st = orc.stats(xb, M, K)
    wk = orc.fc_work(M, K, N)
    assert st.nnz == ref_st.nnz
    assert st.path == orc.decide(M * K, ref_st.nnz, wk.flops_per_byte, wk.macs_eq2, 0.5, 32.0, 0, force)
    ref = orc.fc(xb, M, K, wb, N, bias=bias, act=orc.ACT_GELU)
    got = y.float().cpu().numpy().astype(np.float64)
    assert_close(got, ref, what=f"fused fc {M}x{K}x{N} force={force}")
    assert_occ_equal(yo.to_host(), orc.stats(sp.device_to_bits(y), M, N), "fused fc y_occ")


def test_fused_small_fc_all_zero_and_fp32(sp, ctx):
    """An all-zero input takes the zero-skip path with nothing occupied: the
    output is the epilogue of zero (bias only), written as fp32."""
    M, K, N = 32, 512, 64
    x = torch.zeros(M, K, dtype=torch.bfloat16, device="cuda")
    g = torch.Generator().manual_seed(3)
    wb = synth.to_bf16_bits(torch.randn(N, K, generator=g) / 16)
    wkn = synth.to_bf16_bits(torch.from_numpy(synth.bits_to_f32(wb)).t().contiguous())
    bias = (0.5 * torch.randn(N, generator=g)).numpy().astype(np.float32)
    y = torch.full((M, N), float("nan"), dtype=torch.float32, device="cuda")
    st = sp.sparoa_gemm(ctx, x, sp.bits_to_device(wb).view(N, K), y, W_kn=sp.bits_to_device(wkn).view(K, N),
                        bias=torch.from_numpy(bias).cuda(), host=True)
    assert st.nnz == 0 and st.path == sp.PATH_SKIP
    assert np.array_equal(y.cpu().numpy(), np.broadcast_to(bias, (M, N)))
