"""Parity grid on the GPU: the MLP down projection over token counts, zero
fractions and zero structures, and the dispatch rule exactly at its ties.

The down projection 3072 -> 768 of a ReLU MLP block (the sparsity / intensity
sweep workload) is run through sparoa_gemm at M in {256, 1024, 4096} tokens,
zero fraction rho in {0, 0.5, 0.95}, with unstructured zeros, zeros in 32-channel
blocks per 128-token tile, and whole zero tokens; under the rule and with each
path forced.  The Eq. 1 count is compared with the oracle's in full and bit for
bit, the path with the oracle's rule (Sec. 3: sparsity threshold, then the
intensity threshold) on that count, and the output on a seeded sample of rows
that the oracle computes in fp64.

The tie tests build inputs whose zero count is exactly s_thr * numel, and
thresholds exactly equal to the operator's intensity (FLOPs per input byte, or
the Eq. 2 count in intensity mode 1), and check that the device takes the
oracle's side of each tie: zero-skip at rho == s_thr, dense at intensity ==
c_thr.
"""
import numpy as np
import pytest
import torch

from oracle import oracle as orc
from paper_2511_19457_gb300 import synth
from tests._parity import assert_close

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


@pytest.fixture(scope="module")
def w2(sp):
    wts = synth.mlp_weights(seed=0)
    return wts["w2"], sp.bits_to_device(wts["w2"]).view(768, 3072)


def _f64(t):
    return t.float().cpu().numpy().astype(np.float64)


@pytest.mark.parametrize("force", [0, 1, 2])
@pytest.mark.parametrize("structure", ["unstructured", "block32", "token"])
@pytest.mark.parametrize("rho", [0.0, 0.5, 0.95])
@pytest.mark.parametrize("M", [256, 1024, 4096])
def test_mlp_down_projection_grid(sp, ctx, w2, M, rho, structure, force):
    w_bits, w_dev = w2
    K, N = 3072, 768
    hb = synth.mlp_hidden(M, rho, structure, seed=3 + M)
    h = sp.bits_to_device(hb).view(M, K)
    y = torch.full((M, N), float("nan"), dtype=torch.bfloat16, device="cuda")
    st = sp.sparoa_gemm(ctx, h, w_dev, y, thr=sp.thresholds(force_path=force), host=True)
    ref_st = orc.stats(hb, M, K)
    assert st.nnz == ref_st.nnz
    wk = orc.fc_work(M, K, N)
    want = orc.decide(M * K, ref_st.nnz, wk.flops_per_byte, wk.macs_eq2, 0.5, 32.0, 0, force)
    assert st.path == want
    rows = np.arange(M) if M <= 256 else np.sort(
        np.random.default_rng(M + int(100 * rho)).choice(M, 96, replace=False))
    sub = hb.reshape(M, K)[rows]
    ref = orc.fc(sub, len(rows), K, w_bits, N)
    assert_close(_f64(y)[rows], ref, what=f"M={M} rho={rho} {structure} force={force}")


def _exact_zeros(shape, n_zero, seed):
    """|N(0,1)| + 0.01 everywhere, then exactly n_zero elements set to zero."""
    g = torch.Generator().manual_seed(seed)
    v = torch.randn(*shape, generator=g).abs() + 0.01
    flat = v.reshape(-1)
    idx = torch.randperm(flat.numel(), generator=g)[:n_zero]
    flat[idx] = 0.0
    bits = synth.to_bf16_bits(v)
    assert int(((bits.reshape(-1) & 0x7FFF) == 0).sum()) == n_zero
    return bits


@pytest.mark.parametrize("s_thr", [0.5, 0.375, 0.8125])
@pytest.mark.parametrize("delta", [0, -1])
def test_gemm_sparsity_tie(sp, ctx, s_thr, delta):
    """zeros == s_thr * numel exactly -> zero-skip; one zero fewer -> dense
    (the intensity, N = 64 FLOPs per byte, is above c_thr = 32)."""
    M, K, N = 128, 256, 64
    numel = M * K
    n_zero = int(s_thr * numel) + delta
    xb = _exact_zeros((M, K), n_zero, seed=11)
    g = torch.Generator().manual_seed(12)
    wb = synth.to_bf16_bits(torch.randn(N, K, generator=g) / 16)
    x = sp.bits_to_device(xb).view(M, K)
    w = sp.bits_to_device(wb).view(N, K)
    y = torch.empty(M, N, dtype=torch.bfloat16, device="cuda")
    st = sp.sparoa_gemm(ctx, x, w, y, thr=sp.thresholds(s_thr=s_thr, c_thr=32.0), host=True)
    wk = orc.fc_work(M, K, N)
    want = orc.decide(numel, numel - n_zero, wk.flops_per_byte, wk.macs_eq2, s_thr, 32.0)
    assert want == (orc.PATH_SKIP if delta == 0 else orc.PATH_DENSE)
    assert st.nnz == numel - n_zero and st.path == want
    assert_close(_f64(y), orc.fc(xb, M, K, wb, N), what="tie gemm")


@pytest.mark.parametrize("mode", [0, 1])
@pytest.mark.parametrize("above", [False, True])
def test_gemm_intensity_tie(sp, ctx, mode, above):
    """Intensity exactly c_thr -> dense; the next double above -> zero-skip."""
    M, K, N = 128, 256, 64
    xb = _exact_zeros((M, K), M * K // 4, seed=13)  # rho = 0.25 < s_thr
    g = torch.Generator().manual_seed(14)
    wb = synth.to_bf16_bits(torch.randn(N, K, generator=g) / 16)
    wk = orc.fc_work(M, K, N)
    level = float(wk.flops_per_byte) if mode == 0 else float(wk.macs_eq2)
    c_thr = float(np.nextafter(level, np.inf)) if above else level
    x = sp.bits_to_device(xb).view(M, K)
    w = sp.bits_to_device(wb).view(N, K)
    y = torch.empty(M, N, dtype=torch.bfloat16, device="cuda")
    st = sp.sparoa_gemm(ctx, x, w, y, thr=sp.thresholds(c_thr=c_thr, intensity_mode=mode), host=True)
    want = orc.decide(M * K, M * K - M * K // 4, wk.flops_per_byte, wk.macs_eq2, 0.5, c_thr, mode)
    assert want == (orc.PATH_SKIP if above else orc.PATH_DENSE)
    assert st.path == want
    assert_close(_f64(y), orc.fc(xb, M, K, wb, N), what="intensity tie gemm")


@pytest.mark.parametrize("case", ["rho_tie", "rho_below", "fpb_tie", "fpb_above", "macs_tie", "macs_above"])
def test_conv_ties(sp, ctx, case):
    """The same ties on a 3x3 convolution (64 -> 64, FLOPs per byte 576)."""
    N, H, W, C = 2, 12, 12, 64
    numel = N * H * W * C
    if case == "rho_tie":
        n_zero, s_thr, c_thr, mode = numel // 2, 0.5, 32.0, 0
    elif case == "rho_below":
        n_zero, s_thr, c_thr, mode = numel // 2 - 1, 0.5, 32.0, 0
    else:
        n_zero, s_thr, mode = numel // 4, 0.5, 0 if case.startswith("fpb") else 1
    wk = orc.conv_work(N, H, W, C, C, 3, 3, 1, 1)
    if case.startswith("fpb") or case.startswith("macs"):
        level = float(wk.flops_per_byte) if mode == 0 else float(wk.macs_eq2)
        c_thr = float(np.nextafter(level, np.inf)) if case.endswith("above") else level
    xb = _exact_zeros((N, H, W, C), n_zero, seed=15)
    d = synth.conv_layer(seed=16, N=N, H=H, W=W)
    x = sp.bits_to_device(xb).view(N, H, W, C)
    w = sp.bits_to_device(d["w"]).view(C, 3, 3, C)
    y = torch.empty(N, H, W, C, dtype=torch.bfloat16, device="cuda")
    st = sp.sparoa_conv2d(ctx, x, w, y, stride=1, pad=1, act=sp.ACT_RELU,
                          thr=sp.thresholds(s_thr=s_thr, c_thr=c_thr, intensity_mode=mode), host=True)
    want = orc.decide(numel, numel - n_zero, wk.flops_per_byte, wk.macs_eq2, s_thr, c_thr, mode)
    expect = {"rho_tie": orc.PATH_SKIP, "rho_below": orc.PATH_DENSE, "fpb_tie": orc.PATH_DENSE,
              "fpb_above": orc.PATH_SKIP, "macs_tie": orc.PATH_DENSE, "macs_above": orc.PATH_SKIP}[case]
    assert want == expect
    assert st.nnz == numel - n_zero and st.path == want
    ref = orc.conv2d(xb, N, H, W, C, d["w"], C, 3, 3, 1, 1, act=orc.ACT_RELU)
    assert_close(_f64(y), ref, what=f"conv tie {case}")
