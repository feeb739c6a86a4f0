"""Failure paths on the GPU, made to happen without a GPU fault, trap or hang.

Bounded waits: every wait of the tensor-core kernels on an mbarrier gives up
after a limit of SM cycles.  Here the context's limit is set to about half a
millisecond and the MMA issuer withholds its signal for the first accumulator
of every CTA (a barrier phase that nothing else completes).  The epilogue's
wait runs out, every CTA unwinds (waiting, bounded again, for the copies and
MMAs it already issued), the call that synchronises returns
SPAROA_ERR_TIMEOUT, and the same context then computes the operator correctly.
This is done for the implicit-GEMM kernel (a GEMM and a strided convolution)
and for the 3x3 slab kernel.

Allocation failure: injected on the host; the next workspace allocation of the
context fails, the call returns SPAROA_ERR_OOM, and the next call succeeds.
"""
import numpy as np
import pytest
import torch

from oracle import oracle as orc
from paper_2511_19457_gb300 import synth
from tests._parity import assert_close

pytestmark = pytest.mark.gpu

WAIT_LIMIT = 1 << 20  # SM cycles: about half a millisecond


@pytest.fixture(scope="module")
def sp():
    from paper_2511_19457_gb300 import sparoa
    return sparoa


def _gemm_case(sp, M, K, N, seed):
    g = torch.Generator().manual_seed(seed)
    xb = synth.to_bf16_bits(torch.relu(torch.randn(M, K, generator=g)))
    wb = synth.to_bf16_bits(torch.randn(N, K, generator=g) / np.sqrt(K))
    x = sp.bits_to_device(xb).view(M, K)
    w = sp.bits_to_device(wb).view(N, K)
    ref = orc.fc(xb, M, K, wb, N)

    def run(ctx, force):
        y = torch.full((M, N), float("nan"), dtype=torch.bfloat16, device="cuda")
        st = sp.sparoa_gemm(ctx, x, w, y, thr=sp.thresholds(force_path=force), host=True)
        return st, y
    return run, ref


def _conv_case(sp, N, H, W, C, Co, k, stride, seed):
    d = synth.conv_layer(seed=seed, N=N, H=H, W=W, Cin=C, Cout=Co, k=k, stride=stride, pad=k // 2)
    x = sp.bits_to_device(d["x"]).view(N, H, W, C)
    w = sp.bits_to_device(d["w"]).view(Co, k, k, C)
    Ho, Wo = (H + 2 * (k // 2) - k) // stride + 1, (W + 2 * (k // 2) - k) // stride + 1
    ref = orc.conv2d(d["x"], N, H, W, C, d["w"], Co, k, k, stride, k // 2, act=orc.ACT_RELU)

    def run(ctx, force):
        y = torch.full((N, Ho, Wo, Co), float("nan"), dtype=torch.bfloat16, device="cuda")
        st = sp.sparoa_conv2d(ctx, x, w, y, stride=stride, pad=k // 2, act=sp.ACT_RELU,
                              thr=sp.thresholds(force_path=force), host=True)
        return st, y
    return run, ref


CASES = {
    # implicit-GEMM kernel: several tiles per CTA on 152 SMs
    "gemm": lambda sp: _gemm_case(sp, 4096, 512, 512, 1),
    # implicit-GEMM kernel, strided convolution (4-D TMA boxes)
    "conv3x3s2": lambda sp: _conv_case(sp, 4, 28, 28, 64, 128, 3, 2, 2),
    # 3x3 slab kernel: one and two tiles per CTA
    "conv3x3s1": lambda sp: _conv_case(sp, 8, 56, 56, 64, 64, 3, 1, 3),
}


@pytest.mark.parametrize("name", list(CASES))
@pytest.mark.parametrize("force", [1, 2])
def test_bounded_wait_times_out_and_context_recovers(sp, name, force):
    run, ref = CASES[name](sp)
    ctx = sp.Context(0)
    ctx.set_wait_limit(WAIT_LIMIT)
    ctx.set_fault(1)
    with pytest.raises(sp.SparoaError) as e:
        run(ctx, force)
    assert e.value.status == sp.ERR_TIMEOUT
    # the context (and the device) stay usable: the same call, without the
    # injected fault, computes the operator
    ctx.set_fault(0)
    ctx.set_wait_limit(0)
    st, y = run(ctx, force)
    assert st.path == force
    assert_close(y.float().cpu().numpy().astype(np.float64), ref, what=f"{name} after a timeout")
    ctx.sync()
    ctx.close()


def test_injected_allocation_failure_reports_oom(sp):
    run, ref = _gemm_case(sp, 512, 256, 128, 4)
    ctx = sp.Context(0)
    ctx.set_fault(2)  # the input's occupancy is measured into a workspace grown here
    with pytest.raises(sp.SparoaError) as e:
        run(ctx, 1)
    assert e.value.status == sp.ERR_OOM
    st, y = run(ctx, 1)  # the fault fires once
    assert_close(y.float().cpu().numpy().astype(np.float64), ref, what="gemm after an OOM")
    ctx.close()


def test_hooks_reject_bad_arguments(sp):
    ctx = sp.Context(0)
    assert sp._lib.sparoa_set_wait_limit(ctx.h, -1) == sp.ERR_INVALID_ARG
    assert sp._lib.sparoa_set_fault(ctx.h, 3) == sp.ERR_INVALID_ARG
    assert sp._lib.sparoa_set_fault(None, 0) == sp.ERR_INVALID_ARG
    ctx.close()
