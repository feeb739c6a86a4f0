"""sparoa_run_graph on ResNet-18 and MobileNetV2 topologies against the oracle (GPU).

Teacher forcing: every operator is checked on exactly the bf16 tensor the GPU
fed it (its input read back from the library's workspace), so that Eq. 1
counts, bitmaps and dispatch decisions are compared bit for bit and each
operator's output within the float tolerance.  The chained run (oracle fed only
the graph input) is compared at the end within the float tolerance, or within
twice the network's own sensitivity to one fp32 rounding per operator where
that is larger, with decision flips near the sparsity threshold reported.
"""
import numpy as np
import pytest
import torch

from oracle import oracle as orc
from paper_2511_19457_gb300 import calibrate as cal
from paper_2511_19457_gb300 import synth
from tests._parity import FRO_REL, MAX_REL, assert_close, assert_occ_equal, perturbed_chain_error

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def sp():
    from paper_2511_19457_gb300 import sparoa
    return sparoa


def _run(sp, name, batch, thr=None, table=None):
    ops, xb, shape = getattr(synth, name)(batch=batch, seed=0, thr=thr)
    if table is not None:
        ops = cal.apply(ops, shape, table)
    ctx = sp.Context(0)
    graph = sp.Graph(ops)
    x = sp.bits_to_device(xb).view(*shape)
    last = ops[-1]
    recs = sp.sparoa_run_graph(ctx, graph, x, records=True)
    torch.cuda.synchronize()
    outs, occs = [], []
    for r in recs:
        shp = tuple(int(v) for v in r.out_shape)
        t = sp.view_device(r.output, (int(np.prod(shp)),))
        outs.append((sp.device_to_bits(t), shp))
        occs.append(sp.record_occupancy(r))
    ctx.close()
    return ops, xb, shape, recs, outs, occs


def _teacher_check(sp, ops, xb, shape, recs, outs, occs):
    values = {0: (xb, shape)}
    for i, (bits, shp) in enumerate(outs):
        values[i + 1] = (bits, shp)
    flips = 0
    for i, op in enumerate(ops):
        src = op["input"]
        xin, xs = values[src]
        res = values[op["residual"]][0] if op.get("residual", -1) >= 0 else None
        ref = orc.run_op(op, xin, xs, res)
        r = recs[i]
        assert r.stats.nnz == ref.in_stats.nnz, f"op {i} ({op['kind']}): input nnz"
        assert r.stats.path == ref.path, f"op {i} ({op['kind']}): path {r.stats.path} != {ref.path}"
        if ref.work is not None:
            assert r.stats.flops == ref.work.flops and r.stats.macs_eq2 == ref.work.macs_eq2
        got_bits, got_shape = outs[i]
        assert tuple(got_shape[-1:]) == tuple(ref.out_shape[-1:])
        got = synth.bits_to_f32(got_bits).astype(np.float64).reshape(-1)
        if op["kind"] == "maxpool":
            assert np.array_equal(got, ref.out_f64.reshape(-1)), f"op {i} maxpool"
        else:
            assert_close(got, ref.out_f64, what=f"op {i} ({op['kind']})")
        R = int(np.prod(got_shape[:-1]))
        assert_occ_equal(occs[i], orc.stats(got_bits, R, got_shape[-1]), f"op {i} out occupancy")
    return flips


@pytest.mark.parametrize("name", ["resnet18", "mobilenet_v2"])
def test_graph_teacher_forced(sp, name):
    ops, xb, shape, recs, outs, occs = _run(sp, name, batch=1)
    assert len(recs) == len(ops)
    _teacher_check(sp, ops, xb, shape, recs, outs, occs)
    kinds = [int(r.stats.path) for r in recs]
    assert sp.PATH_DENSE in kinds or sp.PATH_SKIP in kinds
    if name == "mobilenet_v2":
        assert kinds.count(sp.PATH_DEPTHWISE) == 17


def test_graph_batch8_resnet_forced_paths(sp):
    """Both forced paths give the same network output within tolerance."""
    logits = []
    for force in (1, 2):
        ops, xb, shape, recs, outs, occs = _run(sp, "resnet18", batch=8, thr={"force_path": force})
        assert all(int(r.stats.path) in (force, 0) for r in recs)
        logits.append(synth.bits_to_f32(outs[-1][0]).astype(np.float64))
    assert_close(logits[1], logits[0], what="skip vs dense logits")


@pytest.mark.parametrize("name", ["resnet18", "mobilenet_v2"])
def test_graph_chained_end_to_end(sp, name):
    """The oracle fed only the graph input, walking its own values.

    Each operator's output is rounded to bf16 on both sides, so a difference in
    the last fp32 bit before that rounding can move a stored value by one bf16
    step, and the network carries it on.  How far that goes is a property of
    the network, measured here with the oracle alone: its walk with every
    operator output perturbed by at most one fp32 rounding (2^-24 relative).
    The device's chained output must be within the path's float tolerance or,
    where the network's own sensitivity exceeds it, within twice that
    sensitivity.  Operators whose dispatch decision differs between the two
    walks (a zero fraction within rounding of s_thr) are reported, not failed
    on: both paths compute the same operator."""
    ops, xb, shape, recs, outs, occs = _run(sp, name, batch=1)
    ref = orc.run_graph(ops, xb, shape)
    flips = [i for i, (r, o) in enumerate(zip(recs, ref)) if int(r.stats.path) != o.path]
    got = synth.bits_to_f32(outs[-1][0]).astype(np.float64)
    want = ref[-1].out_f64.reshape(-1)
    err = np.abs(got - want)
    s_max, s_fro = perturbed_chain_error(ops, xb, shape, want)
    max_rel, fro_rel = max(MAX_REL, 2 * s_max), max(FRO_REL, 2 * s_fro)
    print(f"{name} chained: max|err|/max|ref| = {err.max() / np.abs(want).max():.3e}, "
          f"rel Frobenius = {np.linalg.norm(got - want) / np.linalg.norm(want):.3e}; "
          f"oracle under one fp32 rounding per op: {s_max:.3e}, {s_fro:.3e}; "
          f"bounds {max_rel:.3e}, {fro_rel:.3e}; decision flips at ops {flips}")
    assert_close(got, want, max_rel=max_rel, fro_rel=fro_rel, what=f"{name} chained logits")


def _mixed_table():
    """Per-kind thresholds spread over always / mid / never zero-skip."""
    kinds = {"conv3x3s1": 0.45, "conv3x3s2": cal.NEVER, "conv1x1s2": 0.0, "conv1x1s1": 0.55,
             "fc_small": 0.0, "gemm": cal.NEVER}
    return {"entries": [{"kind": k, "structure": "unstructured", "flops": 1e9, "s_thr": v}
                        for k, v in kinds.items()]}


@pytest.mark.parametrize("source", ["mixed", "committed"])
@pytest.mark.parametrize("name", ["resnet18", "mobilenet_v2"])
def test_graph_teacher_forced_calibrated(sp, name, source):
    """Per-operator calibrated thresholds: every op's dispatch under its own
    thresholds matches the oracle's, outputs within tolerance."""
    if source == "committed":
        if not __import__("os").path.exists(cal.TABLE_PATH):
            pytest.skip("no calibration table")
        table = cal.load_table()
    else:
        table = _mixed_table()
    ops, xb, shape, recs, outs, occs = _run(sp, name, batch=1, table=table)
    _teacher_check(sp, ops, xb, shape, recs, outs, occs)
    if source == "mixed":
        paths = {int(r.stats.path) for r in recs}
        assert sp.PATH_SKIP in paths and sp.PATH_DENSE in paths
