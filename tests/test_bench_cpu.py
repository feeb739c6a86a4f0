"""bench.py's contract on the host (no GPU): the reference arm's JSON line,
rank handling under a multi-process launch, and the committed per-launch DRAM
traffic entries the roofline object reads."""
import json
import os
import subprocess
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _bench(args, env_extra=None, timeout=300):
    env = dict(os.environ)
    env.update(env_extra or {})
    return subprocess.run([sys.executable, os.path.join(ROOT, "bench.py")] + args, cwd=ROOT, env=env,
                          capture_output=True, text=True, timeout=timeout)


@pytest.fixture(scope="module")
def bench_mod():
    sys.path.insert(0, ROOT)
    import bench
    return bench


def test_reference_arm_line(bench_mod):
    r = _bench(["--impl", "reference", "--steps", "1", "--warmup", "3"])
    assert r.returncode == 0, r.stderr[-2000:]
    lines = [ln for ln in r.stdout.splitlines() if ln.startswith("{")]
    assert len(lines) == 1
    d = json.loads(lines[0])
    assert d["impl"] == "reference"
    assert d["metric"] == bench_mod.METRIC
    assert d["unit"] == "TFLOP/s" and d["higher_is_better"] is True
    assert d["value"] > 0 and d["steps"] == 1 and d["warmup"] == 3 and d["n_gpus"] == 1
    assert d["vs_baseline"] is None and d["data"] == "synthetic"
    assert "workload" in d["config"]
    cb = d["cpu_baseline"]
    assert cb["kind"] == "oracle" and cb["cores"] >= 1 and cb["sample"] and cb["value"] == d["value"]
    e = d["e2e"]
    assert e["value"] == d["value"] and e["unit"] == d["unit"]
    assert e["h2d_bytes_per_step"] == 0 and e["d2h_bytes_per_step"] == 0


def test_reference_arm_other_ranks_do_no_work():
    """Under a multi-process launch only rank 0 runs the oracle and prints."""
    r = _bench(["--impl", "reference", "--gpus", "2", "--steps", "1", "--warmup", "3"],
               {"RANK": "1", "LOCAL_RANK": "1", "WORLD_SIZE": "2"}, timeout=120)
    assert r.returncode == 0, r.stderr[-2000:]
    assert not [ln for ln in r.stdout.splitlines() if ln.startswith("{")]


def test_traffic_entries_name_committed_commands(bench_mod):
    path = os.path.join(ROOT, "profiles", "traffic.json")
    with open(path) as f:
        d = json.load(f)
    assert "conv3_kernel_8x56x56x64" in d  # the default line's dominant kernel
    for key, e in d.items():
        assert key in bench_mod.KERNEL_SOURCES, key
        assert e["dram_bytes_per_launch"] == e["dram_bytes_read"] + e["dram_bytes_write"]
        assert "--clock-control none" in e["capture"] and "python bench.py" in e["capture"]
        assert len(e["kernel_source_sha"]) == 16
        # the hash covers files that exist
        for f in bench_mod.COMMON_SOURCES + bench_mod.KERNEL_SOURCES[key]:
            assert os.path.exists(os.path.join(ROOT, "paper_2511_19457_gb300", "csrc", f)), f
