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
    # ms_per_step is the measured step (one decoder layer's 7 linears); the
    # value scales it to the workload's layers.
    assert line["value"] == pytest.approx(1e3 * line["config"]["batch"] / (line["ms_per_step"] * 2), rel=1e-9)
    assert "x 2 layers" in line["config"]["workload"]


@pytest.mark.parametrize("workload", ["decode", "prefill"])
@pytest.mark.parametrize("schedule", ["dag", "serial", "group", "step"])
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


def _rank_worker(rank, world, port, q):
    import torch
    import torch.distributed as dist
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    sys.path.insert(0, ROOT)
    import bench
    # Rank g took 10 + 5 g seconds for 3 steps of 4 tokens.
    t = bench.max_over_ranks(dist, torch, world, 10.0 + 5.0 * rank, "cpu")
    q.put((rank, t, bench.job_tokens_per_s(4, world, 3, t)))
    dist.destroy_process_group()


def test_job_time_is_the_slowest_rank():
    """Under several ranks the bench times the job by its slowest rank and
    counts every rank's tokens (two gloo processes on the CPU)."""
    import socket
    import torch.multiprocessing as mp
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        port = s.getsockname()[1]
    world = 2
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    procs = [ctx.Process(target=_rank_worker, args=(g, world, port, q)) for g in range(world)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(120)
        assert p.exitcode == 0
    got = sorted(q.get(timeout=10) for _ in range(world))
    for rank, t, v in got:
        assert t == 15.0
        assert v == pytest.approx(4 * 2 * 3 / 15.0)


def test_kernel_bookkeeping_follows_the_dispatch(monkeypatch):
    """The bench names each call's kernel and counts launches from the
    library's dispatch rules: lookup tables up to 4 tokens, the 16-bit-operand
    kernel from 5 to 16, one pass of it for 17-64 tokens on small layers (up
    to 32 tokens below 70 M signs, up to 64 below 20 M), the prefill kernel
    otherwise; layer flags override."""
    sys.path.insert(0, ROOT)
    import bench
    monkeypatch.setattr(bench, "DECODE_KERNEL", "auto")
    assert [bench.decode_kernel_of(b) for b in (1, 2, 4, 5, 8, 16)] == ["lut"] * 3 + ["mma"] * 3
    assert bench.mid_pass_of(4096, 4096, 2028, 17) and bench.mid_pass_of(4096, 4096, 2028, 64)
    assert bench.mid_pass_of(8192, 8192, 4076, 32) and not bench.mid_pass_of(8192, 8192, 4076, 33)
    assert not bench.mid_pass_of(28672, 8192, 6352, 17)
    assert not bench.mid_pass_of(4096, 4096, 2028, 16) and not bench.mid_pass_of(4096, 4096, 2028, 65)
    assert bench.phase_launches(4096, 4096, 2028, 16) == 2
    for forced in ("lut", "tc"):
        monkeypatch.setattr(bench, "DECODE_KERNEL", forced)
        assert not bench.mid_pass_of(4096, 4096, 2028, 17)
        assert bench.decode_kernel_of(1) == forced
    assert bench.phase_launches(4096, 4096, 2028, 8) == 4  # e4m3 kernel: a preparation launch per phase
    monkeypatch.setattr(bench, "DECODE_KERNEL", "mma")
    assert bench.decode_kernel_of(1) == "mma" and bench.mid_pass_of(4096, 4096, 2028, 20)
