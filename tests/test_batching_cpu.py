"""Dynamic batching (Algorithm 2) host logic on synthetic latency / memory models."""
import math

from paper_2511_19457_gb300 import batching as bt


def launch_bound(a=1e-3, b=1e-5):
    # one batch costs a fixed launch-bound part plus a per-image part
    return lambda B: a + b * B


def test_memory_cap_binary_search():
    mem = lambda B: 100 + 10 * B
    assert bt.memory_cap(mem, 1e9) == 512
    assert bt.memory_cap(mem, 100 + 10 * 37) == 37
    assert bt.memory_cap(mem, 100 + 10 * 37 + 9) == 37
    assert bt.memory_cap(mem, 50) == 1  # nothing fits: the smallest batch


def test_launch_bound_grows_and_per_image_latency_falls():
    L = launch_bound()
    tr = bt.dynamic_batch(L, lambda B: 0.0, 1, sparsity=0.0, intensity=0.0)
    assert tr.batch > 16
    # along the gradient steps the per-image latency only falls
    grad = [p for b, l, p, m, n in tr.steps if n in ("initial", "gradient step")]
    assert all(x2 <= x1 * 1.0001 for x1, x2 in zip(grad, grad[1:]))
    # and the stop is where the elasticity has become small
    B = tr.batch
    assert (L(B) / B) <= 1.2 * 1e-5 + 1e-3 / B


def test_flat_per_image_latency_stops_immediately():
    # throughput-bound already at B0: the first probe changes nothing
    tr = bt.dynamic_batch(lambda B: 2e-4 * B, lambda B: 0.0, 8, sparsity=0.0, intensity=0.0)
    assert tr.batch in (8, 16)
    assert len(tr.steps) == 2


def test_memory_constraint_halves():
    mem = lambda B: 1e6 * B
    tr = bt.dynamic_batch(launch_bound(), mem, 4, sparsity=0.0, intensity=0.0, mem_max=2e7)
    assert mem(tr.batch) <= 2e7
    assert any(n == "halved: memory or deadline" for *_, n in tr.steps)


def test_realtime_constraint_halves():
    L = launch_bound(1e-3, 1e-4)
    tr = bt.dynamic_batch(L, lambda B: 0.0, 4, sparsity=0.0, intensity=0.0, t_realtime=3e-3)
    assert L(tr.batch) <= 3e-3
    assert tr.batch <= 20


def test_sparse_input_doubles_up_to_memory():
    mem = lambda B: 1e6 * B
    tr = bt.dynamic_batch(lambda B: 1e-4 * B, mem, 2, sparsity=0.9, intensity=0.0, s_thr=0.5,
                          mem_max=64e6)
    assert any(n == "doubled: sparse input" for *_, n in tr.steps)
    assert tr.batch <= 64
    assert all(b <= 64 for b, *_ in tr.steps if _[-1] == "doubled: sparse input")


def test_intense_input_halves():
    L = launch_bound()
    free = bt.dynamic_batch(L, lambda B: 0.0, 4, sparsity=0.0, intensity=500.0, c_thr=None)
    tr = bt.dynamic_batch(L, lambda B: 0.0, 4, sparsity=0.0, intensity=500.0, c_thr=100.0)
    assert any(n == "halved: intense input" for *_, n in tr.steps)
    assert tr.batch < free.batch
    # below the intensity threshold the rule stays off
    off = bt.dynamic_batch(L, lambda B: 0.0, 4, sparsity=0.0, intensity=50.0, c_thr=100.0)
    assert off.batch == free.batch


def test_bounds_respected_and_trace_serialises():
    tr = bt.dynamic_batch(launch_bound(1.0, 0.0), lambda B: 0.0, 300, sparsity=0.0, intensity=0.0,
                          b_max=512, max_iter=5)
    assert 1 <= tr.batch <= 512
    d = tr.as_dict()
    assert d["batch"] == tr.batch and len(d["steps"]) == len(tr.steps)
    assert all(1 <= s["B"] <= 512 for s in d["steps"])


def test_deadline_bound_does_not_cycle():
    # per-image latency keeps falling, the deadline caps the batch: the search
    # settles below the smallest violating size instead of oscillating
    L = launch_bound(1e-3, 2e-5)
    tr = bt.dynamic_batch(L, lambda B: 0.0, 1, sparsity=0.0, intensity=0.0, t_realtime=2e-3,
                          max_iter=50)
    assert L(tr.batch) <= 2e-3
    assert tr.batch >= 25          # not stuck far below the deadline
    assert len(tr.steps) < 40
