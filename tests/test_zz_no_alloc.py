"""sparoa_gemm_noalloc: the FC operator for callers that cannot allocate (GPU).

Some callers cannot call cudaMalloc: work being recorded into a CUDA graph by
stream capture, plugins living inside another framework's allocator, or loops
with a memory budget fixed at start-up.  sparoa_gemm_noalloc gives them the
same operator with its only scratch (the input's occupancy) in a static
device array.  Here its output, Eq. 1 count and path are checked against
sparoa_gemm on two calls in a row -- a sparse input that takes the zero-skip
path, then a denser, larger one that takes the dense path, so stale contents
of the shared array from the first call would show up in the second -- and an
input too large for the array is rejected.

This file is collected last on purpose: if it fails, a run that stops at the
first failure has already run every other test.
"""
import numpy as np
import pytest
import torch

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


def test_noalloc_matches_gemm_on_two_calls_in_a_row():
    from paper_2511_19457_gb300 import sparoa as sp
    ctx = sp.Context(0)
    cases = [(1, 64, 512, 512, 0.5, True, torch.float32, sp.ACT_NONE, sp.PATH_SKIP),
             (2, 300, 1280, 200, 0.1, False, torch.bfloat16, sp.ACT_RELU, sp.PATH_DENSE)]
    for seed, M, K, N, zp, relu, dt, act, want_path in cases:
        x, w, wkn, bias = _case(seed, M, K, N, zp, relu)
        y_ref = torch.empty(M, N, dtype=dt, device="cuda")
        y_na = torch.full((M, N), float("nan"), dtype=dt, device="cuda")
        st_ref = sp.sparoa_gemm(ctx, x, w, y_ref, W_kn=wkn, bias=bias, act=act, host=True)
        st_na = sp.sparoa_gemm_noalloc(x, w, y_na, W_kn=wkn, bias=bias, act=act, host=True)
        torch.cuda.synchronize()
        assert st_ref.path == want_path
        assert (st_na.nnz, st_na.path, st_na.flops) == (st_ref.nnz, st_ref.path, st_ref.flops)
        assert_close(y_na.float().cpu().numpy(), y_ref.float().cpu().numpy(),
                     what=f"noalloc vs gemm, call seed {seed}")
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
