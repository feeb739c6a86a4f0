"""sparoa_gemm_noalloc: the FC operator for callers that cannot allocate (GPU).

Some callers cannot call cudaMalloc: plugins living inside another framework's
allocator, or loops with a memory budget fixed at start-up.  sparoa_gemm_noalloc gives them the
same operator with its only scratch (the input's occupancy) in a static
device array.  Here its output, Eq. 1 count and path are checked against
sparoa_gemm and against the oracle on several calls in a row -- a sparse input
that takes the zero-skip path, then a denser, larger one that takes the dense
path, then a small one again, so stale contents of the shared array from an
earlier call would show up in a later one -- and an input too large for the
array is rejected.

This file is collected last on purpose: if it fails, a run that stops at the
first failure has already run every other test.
"""
import numpy as np
import pytest
import torch

from oracle import oracle as orc
from paper_2511_19457_gb300 import synth
from tests._parity import assert_close

pytestmark = pytest.mark.gpu


def _case(seed, M, K, N, zero_p, relu):
    g = torch.Generator().manual_seed(seed)
    x = torch.randn(M, K, generator=g)
    if relu:
        x = torch.relu(x)
    x = x * (torch.rand(M, K, generator=g) >= zero_p).to(torch.float32)
    w = torch.randn(N, K, generator=g) / np.sqrt(K)
    bias = 0.1 * torch.randn(N, generator=g)
    return (x.to(torch.bfloat16).cuda(), w.to(torch.bfloat16).cuda(),
            w.t().contiguous().to(torch.bfloat16).cuda(), bias.cuda())


def _host_bits(t):
    return t.cpu().view(torch.int16).numpy().view(np.uint16)


def test_noalloc_matches_gemm_on_two_calls_in_a_row():
    """Consecutive calls share the static array: a sparse small FC (zero-skip),
    a larger dense one, then a K = 64 one (whose row bitmaps the statistics
    write whole while the rest of the array still holds the larger call's
    contents), a GELU epilogue, and both forced paths.  Each is compared with
    sparoa_gemm (output, Eq. 1 count, path) and with the oracle."""
    from paper_2511_19457_gb300 import sparoa as sp
    ctx = sp.Context(0)
    cases = [(1, 64, 512, 512, 0.5, True, torch.float32, sp.ACT_NONE, 0, sp.PATH_SKIP),
             (2, 300, 1280, 200, 0.1, False, torch.bfloat16, sp.ACT_RELU, 0, sp.PATH_DENSE),
             (3, 100, 64, 64, 0.6, True, torch.bfloat16, sp.ACT_NONE, 0, sp.PATH_SKIP),
             (4, 96, 256, 128, 0.2, False, torch.bfloat16, sp.ACT_GELU, 0, sp.PATH_DENSE),
             (5, 100, 64, 64, 0.1, True, torch.bfloat16, sp.ACT_RELU, 2, sp.PATH_SKIP),
             (6, 200, 128, 64, 0.7, True, torch.float32, sp.ACT_NONE, 1, sp.PATH_DENSE)]
    for seed, M, K, N, zp, relu, dt, act, force, want_path in cases:
        x, w, wkn, bias = _case(seed, M, K, N, zp, relu)
        thr = sp.thresholds(force_path=force)
        y_ref = torch.empty(M, N, dtype=dt, device="cuda")
        y_na = torch.full((M, N), float("nan"), dtype=dt, device="cuda")
        st_ref = sp.sparoa_gemm(ctx, x, w, y_ref, W_kn=wkn, bias=bias, act=act, thr=thr, host=True)
        st_na = sp.sparoa_gemm_noalloc(x, w, y_na, W_kn=wkn, bias=bias, act=act, thr=thr, host=True)
        torch.cuda.synchronize()
        assert st_ref.path == want_path
        assert (st_na.nnz, st_na.path, st_na.flops) == (st_ref.nnz, st_ref.path, st_ref.flops)
        got = y_na.float().cpu().numpy()
        assert_close(got, y_ref.float().cpu().numpy(), what=f"noalloc vs gemm, call seed {seed}")
        xb, wb = _host_bits(x), _host_bits(w)
        assert st_na.nnz == orc.stats(xb, M, K).nnz
        ref = orc.fc(xb, M, K, wb, N, bias=bias.cpu().numpy(), act=act)
        if dt == torch.bfloat16:
            ref = synth.bits_to_f32(orc.f64_to_bf16(ref)).astype(np.float64)
        assert_close(got, ref, what=f"noalloc vs oracle, call seed {seed}")
    ctx.close()


def test_noalloc_rejects_inputs_beyond_the_static_array():
    from paper_2511_19457_gb300 import sparoa as sp
    x = torch.zeros(8, 64, dtype=torch.bfloat16, device="cuda")
    w = torch.zeros(64, 64, dtype=torch.bfloat16, device="cuda")
    y = torch.zeros(8, 64, dtype=torch.bfloat16, device="cuda")
    big_m = 1 << 20   # occupancy of [2^20, 64]: 8 MiB of row bitmap > 4 MiB array
    rc = sp._lib.sparoa_gemm_noalloc(None, sp._ptr(x), big_m, 64, sp._ptr(w), None, 64, None, None,
                                     sp._ptr(y), sp.BF16, None)
    assert rc == sp.ERR_UNSUPPORTED
