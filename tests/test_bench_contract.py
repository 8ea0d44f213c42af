"""bench.py's output contract, checked on the CPU: the reference arm (the
FP64 oracle timed on the host cores) prints one JSON line with the keys the
measurement needs, its value consistent with its step time, and every
workload and schedule has a configuration description."""
import json
import os
import subprocess
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
KEYS = ("impl", "metric", "value", "unit", "n_gpus", "steps", "warmup", "ms_per_step", "higher_is_better",
        "scaling", "vs_baseline", "dtype", "data", "config", "cpu_baseline", "e2e")


def test_reference_arm_line():
    out = subprocess.run([sys.executable, "bench.py", "--impl", "reference", "--steps", "1", "--warmup", "0",
                          "--layers", "2"], cwd=ROOT, capture_output=True, text=True, timeout=600)
    assert out.returncode == 0, out.stderr
    line = json.loads(out.stdout.strip().splitlines()[-1])
    for k in KEYS:
        assert k in line, k
    assert line["impl"] == "reference" and line["value"] > 0 and line["unit"] == "tokens/s"
    assert line["higher_is_better"] is True and line["vs_baseline"] is None
    cb = line["cpu_baseline"]
    assert cb["kind"] == "oracle" and cb["cores"] >= 1 and cb["value"] == line["value"]
    assert "1/2 of the workload" in cb["sample"]
    e2e = line["e2e"]
    assert e2e["value"] == line["value"] and e2e["h2d_bytes_per_step"] == 0 and e2e["d2h_bytes_per_step"] == 0
    # tokens per step / step time: one token per step over the 2 layers timed.
    assert line["value"] == pytest.approx(1e3 * line["config"]["batch"] / line["ms_per_step"], rel=1e-9)
    assert "x 2 layers" in line["config"]["workload"]


@pytest.mark.parametrize("workload", ["decode", "prefill"])
@pytest.mark.parametrize("schedule", ["dag", "serial", "group"])
def test_config_names_the_schedule(monkeypatch, workload, schedule):
    sys.path.insert(0, ROOT)
    import bench
    monkeypatch.setattr(sys, "argv", ["bench.py", "--workload", workload, "--schedule", schedule])
    args = bench.parse()
    b = bench.resolve_workload(args)
    cfg = bench.config_dict(args)
    assert bench.SCHEDULES[schedule] in cfg["workload"]
    if workload == "prefill":
        assert b == 2048 and args.layers == 4 and cfg["tokens"] == 2048
    else:
        assert b == 1 and args.layers == bench.LAYERS and cfg["batch"] == 1


def test_workload_bounds(monkeypatch):
    sys.path.insert(0, ROOT)
    import bench
    for argv in (["--batch", "17"], ["--batch", "0"], ["--workload", "prefill", "--tokens", "16"]):
        monkeypatch.setattr(sys, "argv", ["bench.py"] + argv)
        with pytest.raises(SystemExit):
            bench.resolve_workload(bench.parse())
