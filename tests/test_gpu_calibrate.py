"""The threshold calibration's measurement loop on the GPU (small grid)."""
import pytest

from paper_2511_19457_gb300 import calibrate as cal

pytestmark = pytest.mark.gpu


def test_calibrate_small_grid():
    from paper_2511_19457_gb300 import sparoa as sp
    ctx = sp.Context(0)
    specs = (("fc", (64, 512, 512)), ("fc", (300, 256, 128)), ("conv", (2, 16, 16, 64, 64, 3, 1, 1)),
             ("conv", (2, 16, 16, 32, 64, 1, 2, 0)))
    t = cal.calibrate(ctx, specs=specs, rhos=(0.0, 0.95), structures=("block",), max_sets=2, replays=2)
    ctx.close()
    assert len(t["entries"]) == len(specs)
    for e, (op, shape) in zip(t["entries"], specs):
        assert e["op"] == op and tuple(e["shape"]) == shape and e["structure"] == "block"
        assert len(e["dense_us"]) == len(e["skip_us"]) == 2
        assert all(v > 0 for v in e["dense_us"] + e["skip_us"])
        assert e["measured_rho"][0] == 0.0
        assert 0.6 < e["measured_rho"][1] <= 1.0  # few block units: a loose bound
        assert e["s_thr"] == cal.crossover(e["rho"], e["dense_us"], e["skip_us"])
