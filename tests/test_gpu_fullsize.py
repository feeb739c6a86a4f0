"""Parity at the graph workloads' full sizes, in the launch configuration the
bench times: ResNet-18, MobileNetV2 and ViT-B/16 at batch 32, each one
sparoa_run_graph over the whole batch (GPU).

Every operator is teacher-forced on the bf16 tensor the GPU fed it.  Integer
results are compared in full and bit for bit: the input's Eq. 1 count, the
dispatch decision, the Eq. 2 work and the output's occupancy block.  Float
outputs are compared on a seeded sample that the oracle computes one output at
a time: a conv output from the k x k input window it depends on (convolution
is local; the padding is written into the window as zeros), FC and layer-norm
outputs on sampled rows, attention on one sampled image; pools, batch norm,
the token sequence and token selection in full (the oracle is fast there).
"""
import numpy as np
import pytest

from oracle import oracle as orc
from paper_2511_19457_gb300 import synth
from tests._parity import assert_close, assert_occ_equal

pytestmark = pytest.mark.gpu

SAMPLES = 24  # sampled outputs (conv positions, FC / layer-norm rows) per operator


@pytest.fixture(scope="module")
def sp():
    from paper_2511_19457_gb300 import sparoa
    return sparoa


def _window(xin, shape, n, oh, ow, k, s, p):
    """The k x k input window of output (n, oh, ow), zeros (+0.0) where it
    reaches into the padding."""
    N, H, W, C = shape
    x = xin.reshape(N, H, W, C)
    win = np.zeros((1, k, k, C), dtype=np.uint16)
    for dy in range(k):
        iy = oh * s - p + dy
        if 0 <= iy < H:
            for dx in range(k):
                ix = ow * s - p + dx
                if 0 <= ix < W:
                    win[0, dy, dx] = x[n, iy, ix]
    return win


def _expected_path(op, xs, nnz):
    thr = op.get("thr", {})
    args = (thr.get("s_thr", 0.5), thr.get("c_thr", 32.0), thr.get("intensity_mode", 0),
            thr.get("force_path", 0))
    if op["kind"] == "conv":
        N, H, W, C = xs
        if op.get("groups", 1) != 1:
            return orc.PATH_DEPTHWISE, None
        wk = orc.conv_work(N, H, W, C, op["cout"], op["k"], op["k"], op["stride"], op["pad"], 1)
        return orc.decide(N * H * W * C, nnz, wk.flops_per_byte, wk.macs_eq2, *args), wk
    if op["kind"] == "fc":
        M, K = xs[0], int(np.prod(xs[1:]))
        wk = orc.fc_work(M, K, op["cout"])
        return orc.decide(M * K, nnz, wk.flops_per_byte, wk.macs_eq2, *args), wk
    return orc.PATH_NONE, None


def _sampled_outputs(op, xin, xs, res, got, gshape, rng):
    """(GPU values, oracle values) on this operator's sample."""
    kind = op["kind"]
    eps = op.get("eps", 1e-5)
    act = op.get("act", orc.ACT_NONE)
    if kind == "conv":
        N, Ho, Wo, Co = gshape
        k, s, p, g = op["k"], op["stride"], op["pad"], op.get("groups", 1)
        y = got.reshape(N, Ho, Wo, Co)
        r4 = None if res is None else res.reshape(N, Ho, Wo, Co)
        gots, refs = [], []
        for m in rng.integers(0, N * Ho * Wo, SAMPLES):
            n, rem = divmod(int(m), Ho * Wo)
            oh, ow = divmod(rem, Wo)
            win = _window(xin, xs, n, oh, ow, k, s, p)
            rb = None if r4 is None else np.ascontiguousarray(r4[n, oh, ow])
            ref = orc.conv2d(win, 1, k, k, xs[3], op["w"], Co, k, k, 1, 0, g, op.get("bias"),
                             op.get("bn"), eps, rb, act)
            gots.append(y[n, oh, ow])
            refs.append(ref.reshape(-1))
        return np.concatenate(gots), np.concatenate(refs)
    if kind == "fc":
        M, K = xs[0], int(np.prod(xs[1:]))
        rows = np.sort(rng.choice(M, min(M, SAMPLES), replace=False))
        sub = np.ascontiguousarray(xin.reshape(M, K)[rows])
        rb = None if res is None else np.ascontiguousarray(res.reshape(M, -1)[rows])
        ref = orc.fc(sub, len(rows), K, op["w"], op["cout"], op.get("bias"), op.get("bn"), eps, rb, act)
        return got.reshape(M, -1)[rows], ref
    if kind == "layernorm":
        C = xs[-1]
        R = int(np.prod(xs[:-1]))
        rows = np.sort(rng.choice(R, min(R, SAMPLES), replace=False))
        sub = np.ascontiguousarray(xin.reshape(R, C)[rows])
        ref = orc.layernorm(sub, len(rows), C, op.get("gamma_beta"), op.get("eps", 1e-6))
        return got.reshape(R, C)[rows], ref
    if kind == "attention":
        N, H, W, C3 = xs
        T, heads = H * W, op["heads"]
        n = int(rng.integers(0, N))
        one = np.ascontiguousarray(xin.reshape(N, T, C3)[n])
        ref = orc.attention(one, 1, T, heads, C3 // 3 // heads)
        return got.reshape(N, T, -1)[n], ref
    ref = orc.run_op(op, xin, xs, res).out_f64
    return got, ref


@pytest.mark.parametrize("name", ["resnet18", "mobilenet_v2", "vit"])
def test_graph_batch32_sampled(sp, name):
    from tests.test_gpu_graph import _run
    ops, xb, shape, recs, outs, occs = _run(sp, name, batch=32)
    assert len(recs) == len(ops)
    rng = np.random.default_rng(32)
    values = {0: (xb, tuple(shape))}
    for i, (bits, shp) in enumerate(outs):
        values[i + 1] = (bits, tuple(shp))
    for i, op in enumerate(ops):
        xin, xs = values[op["input"]]
        res = values[op["residual"]][0] if op.get("residual", -1) >= 0 else None
        r = recs[i]
        what = f"{name} op {i} ({op['kind']})"
        nnz = orc.stats(xin, int(np.prod(xs[:-1])), xs[-1]).nnz
        assert r.stats.nnz == nnz, f"{what}: input nnz"
        path, wk = _expected_path(op, xs, nnz)
        if op["kind"] in ("conv", "fc"):
            assert r.stats.path == path, f"{what}: path {r.stats.path} != {path}"
        if wk is not None:
            assert r.stats.flops == wk.flops and r.stats.macs_eq2 == wk.macs_eq2, f"{what}: work"
        got_bits, gshape = outs[i]
        got = synth.bits_to_f32(got_bits).astype(np.float64)
        g, ref = _sampled_outputs(op, xin, xs, res, got, gshape, rng)
        if op["kind"] == "maxpool":
            assert np.array_equal(np.asarray(g).reshape(-1), ref.reshape(-1)), what
        else:
            assert_close(g, ref, what=what)
        R = int(np.prod(gshape[:-1]))
        assert_occ_equal(occs[i], orc.stats(got_bits, R, gshape[-1]), f"{what}: output occupancy")
