"""A 3x3 convolution that measures its own input, without a host record.

Without x_occ, sparoa_conv2d launches a small clear of the input's counters
and block masks, the statistics kernel (Eq. 1 count and masks of x; it also
zeroes the output's occupancy block, and reads x before its
griddepcontrol.wait) and the conv kernel (weights, first slab and column
affine loaded before its wait; the Sec. 3 rule on the device).  Nothing is
carried between calls, so repeated calls, calls of different shapes and
CUDA-graph replays of any number of calls all see the same counts.

Checked against the oracle: the output (float tolerance), the output's
occupancy (bit for bit, on the bf16 output the GPU produced), and the path
the device recorded against the oracle's rule on the input's count -- at and
either side of the sparsity tie, and on an all-zero input.  The same calls
with a host record (counts accumulated after a clear launch) give the same
bits.
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


def _bits(t):
    return t.contiguous().view(torch.int16).cpu().numpy().view(np.uint16).reshape(-1)


def _exact_zeros(shape, n_zero, seed):
    g = torch.Generator().manual_seed(seed)
    v = torch.randn(*shape, generator=g).abs() + 0.01
    flat = v.reshape(-1)
    idx = torch.randperm(flat.numel(), generator=g)[:n_zero]
    flat[idx] = 0.0
    return synth.to_bf16_bits(v)


class Case:
    def __init__(self, sp, N, H, W, xb, seed):
        C = 64
        self.N, self.H, self.W, self.C = N, H, W, C
        d = synth.conv_layer(seed=seed, N=N, H=H, W=W)
        self.xb, self.wb, self.bn = xb, d["w"], d["bn"]
        self.x = sp.bits_to_device(xb).view(N, H, W, C)
        self.w = sp.bits_to_device(self.wb).view(C, 3, 3, C)
        self.bn_dev = torch.from_numpy(self.bn).cuda()
        self.ref = orc.conv2d(xb, N, H, W, C, self.wb, C, 3, 3, 1, 1, bn=self.bn, act=orc.ACT_RELU)
        self.numel = N * H * W * C
        self.nnz = orc.stats(xb, N * H * W, C).nnz
        self.wk = orc.conv_work(N, H, W, C, C, 3, 3, 1, 1)

    def want(self, s_thr=0.5, c_thr=32.0, force=0):
        return orc.decide(self.numel, self.nnz, self.wk.flops_per_byte, self.wk.macs_eq2, s_thr, c_thr,
                          0, force)

    def run(self, sp, ctx, thr, host=False):
        y = torch.full((self.N, self.H, self.W, self.C), float("nan"), dtype=torch.bfloat16, device="cuda")
        yo = sp.OccupancyBuffer(self.N * self.H * self.W, self.C)
        yo.buf.fill_(0xA5)  # garbage: the call zeroes the block itself
        st = sp.sparoa_conv2d(ctx, self.x, self.w, y, stride=1, pad=1, bn=self.bn_dev, act=sp.ACT_RELU,
                              thr=thr, y_occ=yo, host=host)
        return st, y, yo

    def check(self, y, yo, what):
        assert_close(y.float().cpu().numpy().astype(np.float64), self.ref, what=what)
        yb = _bits(y)
        assert_occ_equal(yo.to_host(), orc.stats(yb, self.N * self.H * self.W, self.C), what=what)


def _random_case(sp, N, H, W, seed):
    d = synth.conv_layer(seed=seed, N=N, H=H, W=W)
    return Case(sp, N, H, W, d["x"], seed)


@pytest.mark.parametrize("shape", [(8, 56, 56), (3, 17, 23), (1, 5, 7)])
@pytest.mark.parametrize("force", [0, 1, 2])
def test_measured_conv_matches_oracle(sp, ctx, shape, force):
    c = _random_case(sp, *shape, seed=40 + shape[1])
    thr = sp.thresholds(force_path=force)
    _, y, yo = c.run(sp, ctx, thr)
    assert ctx.last_path() == c.want(force=force)
    c.check(y, yo, f"measured conv {shape} force {force}")
    # with a host record: the accumulated counts, the same output bits
    st, y2, yo2 = c.run(sp, ctx, thr, host=True)
    assert st.nnz == c.nnz and st.path == c.want(force=force)
    assert np.array_equal(_bits(y), _bits(y2))


@pytest.mark.parametrize("delta", [0, -1, 1])
def test_measured_conv_sparsity_tie(sp, ctx, delta):
    """zeros == s_thr * numel -> zero-skip; one fewer -> dense; one more -> zero-skip."""
    N, H, W, C = 2, 12, 12, 64
    numel = N * H * W * C
    c = Case(sp, N, H, W, _exact_zeros((N, H, W, C), numel // 2 + delta, seed=17), seed=18)
    assert c.nnz == numel - (numel // 2 + delta)
    _, y, yo = c.run(sp, ctx, sp.thresholds())
    want = c.want()
    assert want == (orc.PATH_DENSE if delta < 0 else orc.PATH_SKIP)
    assert ctx.last_path() == want
    c.check(y, yo, f"tie {delta}")


def test_measured_conv_all_zero_input(sp, ctx):
    N, H, W, C = 2, 9, 9, 64
    c = Case(sp, N, H, W, np.zeros(N * H * W * C, dtype=np.uint16), seed=19)
    _, y, yo = c.run(sp, ctx, sp.thresholds())
    assert ctx.last_path() == orc.PATH_SKIP
    c.check(y, yo, "all-zero input")


def test_measured_conv_repeated_and_mixed_shapes(sp, ctx):
    """Nothing carries over between calls: repeated calls and a change of shape."""
    big = _random_case(sp, 8, 56, 56, seed=21)
    small = _random_case(sp, 3, 17, 23, seed=22)
    for c in (big, big, small, big, small, small):
        _, y, yo = c.run(sp, ctx, sp.thresholds())
        assert ctx.last_path() == c.want()
        c.check(y, yo, f"repeated {c.N}x{c.H}x{c.W}")


@pytest.mark.parametrize("calls", [1, 3])
def test_measured_conv_graph_replays(sp, ctx, calls):
    """A CUDA graph of an odd number of measuring calls, replayed: every replay
    gives the oracle's output, occupancy and path."""
    c = _random_case(sp, 4, 28, 28, seed=23)
    thr = sp.thresholds()
    ys = [torch.empty(c.N, c.H, c.W, c.C, dtype=torch.bfloat16, device="cuda") for _ in range(calls)]
    yos = [sp.OccupancyBuffer(c.N * c.H * c.W, c.C) for _ in range(calls)]

    def body():
        for j in range(calls):
            sp.sparoa_conv2d(ctx, c.x, c.w, ys[j], stride=1, pad=1, bn=c.bn_dev, act=sp.ACT_RELU, thr=thr,
                             y_occ=yos[j])

    s = torch.cuda.Stream()
    s.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(s):
        body()
    torch.cuda.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=s):
        body()
    for rep in range(3):
        for j in range(calls):
            ys[j].fill_(float("nan"))
            yos[j].buf.fill_(0xA5)
        g.replay()
        torch.cuda.synchronize()
        assert ctx.last_path() == c.want()
        for j in range(calls):
            c.check(ys[j], yos[j], f"graph replay {rep} call {j}")
