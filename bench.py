"""Benchmark: AF1 binary-factorized linears (decode path by default).

Workload (default): a 32-layer LLaMA-3-8B-shaped linear stack, the seven
linears of each decoder layer (q, k, v, o, gate, up, down) with HiSA-like
ranks: each matrix's exact 1.0-BPW rank times a seeded factor in [0.7, 1.3],
renormalised so the whole stack stays within 1.0 bit per weight. Distinct
seeded synthetic weights (about 0.87 GB of packed signs per step, far above
the 129 MB L2, so no flush is needed). One step is one decode token (batch
1 by default) through all 224 linears through af1_linear_forward on the
decoder's dependency DAG, replayed as a CUDA graph. `--ranks uniform` uses
every matrix's 1.0-BPW rank instead.

`--workload prefill` times the tensor-core prefill path instead: the same
seven linears over 4 layers at 2048 tokens per call (1 % outlier channels),
reported against the tensor roofline.

Prints one JSON line. `--impl reference` times the CPU FP64 oracle instead
(the reference arm of this paper-only build), on a bounded sample per step.
"""
from __future__ import annotations

import argparse
import json
import os
import subprocess
import sys
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

NCORES = len(os.sched_getaffinity(0))
for _v in ("OPENBLAS_NUM_THREADS", "OMP_NUM_THREADS", "MKL_NUM_THREADS"):
    os.environ.setdefault(_v, str(NCORES))

import numpy as np  # noqa: E402

METRIC = "tokens/s and us/layer for binary-factorized linear (AF1, 1.0 BPW); % of HBM roofline"
LAYERS = 32
# Measured DRAM traffic of one layer's seven decode calls at one token (bytes;
# ncu, profiles/lut_kernel_llama3_8b_b1.md): 1.026 x the algorithmic bytes.
DECODE_TRAFFIC_B1_PER_LAYER = 28145408
# The same for the HiSA-rank stack on the DAG schedule: DRAM bytes (read +
# write) of one step's 84 lookup-table launches over 6 layers, divided by that
# step's algorithmic bytes (ncu, profiles/lut_kernel_llama3_8b_hisa_b1.md);
# a full step's traffic is this ratio times its algorithmic bytes.
DECODE_TRAFFIC_RATIO_HISA_B1 = 170377216 / 164560648
# The same on the grouped schedule (q|k|v and gate|up as one multi-layer call
# each): ncu, profiles/lut_kernel_llama3_8b_hisa_b1_group.md.
DECODE_TRAFFIC_RATIO_HISA_B1_GROUP = 169402880 / 164560648
DECODE_KERNEL = "auto"  # set from --decode-kernel / --tc-decode


def parse():
    p = argparse.ArgumentParser()
    p.add_argument("--gpus", type=int, default=1)
    p.add_argument("--steps", type=int, default=50)
    p.add_argument("--warmup", type=int, default=5)
    p.add_argument("--batch", type=int, default=1, help="decode tokens per step (1..16)")
    p.add_argument("--impl", choices=["af1", "reference"], default="af1")
    p.add_argument("--layers", type=int, default=LAYERS)
    p.add_argument("--no-dense", action="store_true", help="skip the dense BF16 baseline")
    p.add_argument("--no-cpu", action="store_true", help="skip the CPU oracle baseline")
    p.add_argument("--workload", choices=["decode", "prefill"], default="decode",
                   help="decode: config 1 (1-16 tokens); prefill: config 2 (2048 tokens, tensor cores)")
    p.add_argument("--tokens", type=int, default=2048, help="prefill tokens per call")
    p.add_argument("--no-graph", action="store_true", help="eager launches instead of a CUDA graph (for profilers)")
    p.add_argument("--schedule", choices=["dag", "serial", "group", "step"], default=None,
                   help="dag: a decoder layer's independent linears (q/k/v, gate/up) on parallel streams; "
                        "serial: all 7 linears chained on one stream; group: q|k|v and gate|up as one "
                        "af1_linear_forward_multi call each (shared input), one stream; step: the whole step "
                        "as one persistent launch (af1_step_run) with the DAG's level order. Default: group for "
                        "decode passes of 1-2 tokens, dag otherwise (the faster of the two measured on GB300: "
                        "1 token 1.32 vs 1.43 ms per step, 16 tokens 6.39 vs 5.30)")
    p.add_argument("--ranks", choices=["hisa", "uniform"], default="hisa",
                   help="decode stack ranks: hisa = 1.0-BPW rank x U(0.7, 1.3), renormalised to 1.0 BPW over the "
                        "stack (the default workload); uniform = every matrix at its 1.0-BPW rank")
    p.add_argument("--no-sweep", action="store_true",
                   help="skip the per-shape sweep (LLaMA-3-8B at 1/4/16 tokens, 70B shapes at 1/8/64/512)")
    p.add_argument("--no-stack", action="store_true", help="skip the 32-layer stack with HiSA-like ranks")
    p.add_argument("--shape", default=None, metavar="MxN",
                   help="time one linear of this shape (1.0-BPW rank) at --batch tokens instead of the stack: "
                        "--steps calls rotating over copies larger than L2; prints one JSON line (per-shape "
                        "measurement and profiling, e.g. with --no-graph under ncu)")
    p.add_argument("--tc-decode", action="store_true",
                   help="create layers with AF1_FLAG_TC_DECODE (the e4m3 tensor-core decode kernel); "
                        "same as --decode-kernel tc")
    p.add_argument("--decode-kernel", choices=["auto", "lut", "mma", "tc"], default="auto",
                   help="decode kernel of the layers: auto (the library's dispatch: lookup tables below 4 tokens, "
                        "16-bit-operand tensor cores from 4), lut (AF1_FLAG_LUT_DECODE), mma (AF1_FLAG_MMA_DECODE), "
                        "tc (AF1_FLAG_TC_DECODE)")
    a = p.parse_args()
    if a.schedule is None:
        a.schedule = "group" if (a.workload == "decode" and a.batch <= 2) else "dag"
    return a


def workload_ranks(args, rank_fn=None, bits_fn=None):
    """Rank of every linear of the stack, in model order (7 per layer)."""
    import synth
    if rank_fn is None:
        import paper_2609_06161_gb300 as P
        rank_fn = P.rank_for_budget
    mn = [(m, n) for _ in range(args.layers) for (_nm, m, n) in synth.LLAMA3_8B_LINEARS]
    if args.workload == "decode" and args.ranks == "hisa":
        return hisa_ranks(mn, rank_fn=rank_fn, bits_fn=bits_fn)
    return [int(rank_fn(m, n)) for (m, n) in mn]


def shapes(rank_fn=None):
    """The seven LLaMA-3-8B decoder linears at their exact 1.0-BPW ranks.
    rank_fn defaults to the library's rank rule; the oracle legs pass the
    oracle's."""
    import synth
    if rank_fn is None:
        import paper_2609_06161_gb300 as P
        rank_fn = P.rank_for_budget
    return [(name, m, n, int(rank_fn(m, n))) for name, m, n in synth.LLAMA3_8B_LINEARS]


def oracle_shapes():
    from oracle import af1_oracle as O
    return shapes(lambda m, n: O.rank_for_budget(m, n, 1))


def hisa_ranks(mn, seed=3, rank_fn=None, bits_fn=None):
    """HiSA-like rank allocation over the matrices `mn` = [(m, n), ...]: each
    1.0-BPW rank scaled by a seeded factor in [0.7, 1.3], then renormalised
    so that the total storage stays within 1.0 bit per weight: one common
    factor, floor, then +1 steps in a seeded order while the budget holds
    (slack below one rank step)."""
    import math
    import synth
    if rank_fn is None or bits_fn is None:
        import paper_2609_06161_gb300 as P
        rank_fn = rank_fn or P.rank_for_budget
        bits_fn = bits_fn or P.storage_bits
    base = [rank_fn(m, n) for (m, n) in mn]
    f, order = synth.hisa_rank_factors(seed, len(mn))
    drawn = [max(1, int(round(b * fi))) for b, fi in zip(base, f)]
    budget = sum(m * n for (m, n) in mn)
    fixed = sum(bits_fn(m, n, 1) - (m + n + 16) for (m, n) in mn)  # 16 (m + n) per matrix
    per = sum(r * (m + n + 16) for r, (m, n) in zip(drawn, mn))
    c = (budget - fixed) / per
    ranks = [max(1, math.floor(c * r)) for r in drawn]
    total = sum(bits_fn(m, n, r) for r, (m, n) in zip(ranks, mn))
    while total > budget:  # floor of a positive factor cannot overshoot; kept as a guard
        i = max(range(len(ranks)), key=lambda j: ranks[j])
        total -= mn[i][0] + mn[i][1] + 16
        ranks[i] -= 1
    grew = True
    while grew:
        grew = False
        for i in order:
            step = mn[i][0] + mn[i][1] + 16
            if total + step <= budget:
                ranks[i] += 1
                total += step
                grew = True
    return ranks


def algorithmic_bytes(m, n, r, b):
    """Logical packed sign bits / 8 + FP16 scales + FP16 x and y."""
    return r * (m + n) // 8 + 2 * (m + n + r) + 2 * b * n + 2 * b * m


def dist_env():
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return world, rank, local


def max_over_ranks(dist, torch, world, value, device):
    """The job's time: the largest of the ranks' times (every rank gets it)."""
    t = torch.tensor([float(value)], dtype=torch.float64, device=device)
    if world > 1:
        dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def job_tokens_per_s(tokens_per_rank_step, world, steps, seconds):
    """Whole-job throughput: every rank's tokens over the slowest rank's time."""
    return tokens_per_rank_step * world * steps / seconds


# ---------------------------------------------------------------------------
# CPU oracle timing (cpu_baseline and the reference arm)
# ---------------------------------------------------------------------------

def oracle_ranks(args):
    """The stack's ranks by the oracle's rank rule (the host legs need no GPU
    library)."""
    from oracle import af1_oracle as O
    return workload_ranks(args, rank_fn=lambda m, n: O.rank_for_budget(m, n, 1), bits_fn=O.storage_bits)


def oracle_layer_sample(batch, ranks7, seed_base=0):
    """The 7 linears of one decoder layer (ranks ranks7), as canonical packed words."""
    import synth
    data = []
    for i, (name, m, n) in enumerate(synth.LLAMA3_8B_LINEARS):
        r = ranks7[i]
        d = synth.layer_words(seed_base + i, m, n, r, batch)
        data.append((name, m, n, r, d))
    return data


def time_oracle_layer(data):
    from oracle import af1_oracle as O
    t0 = time.perf_counter()
    for (_name, m, n, r, d) in data:
        O.forward_from_packed(d["Uw"], d["Vw"], d["a"], d["s"], d["b"], d["x"], m, n, r)
    return time.perf_counter() - t0


def resolve_workload(args):
    """Tokens per call of the workload; the prefill workload defaults to 4
    layers (a step of 28 calls at 2048 tokens)."""
    if args.workload == "prefill":
        if args.tokens <= 16:
            raise SystemExit("--tokens must be > 16 for the prefill path")
        if args.layers == LAYERS:
            args.layers = 4
        return args.tokens
    if not 1 <= args.batch <= 16:
        raise SystemExit("--batch must be in 1..16 for the decode path")
    return args.batch


def cpu_baseline(batch, layers, ranks7, min_seconds=10.0):
    data = oracle_layer_sample(batch, ranks7)
    times = []
    t_start = time.perf_counter()
    while True:
        times.append(time_oracle_layer(data))
        if time.perf_counter() - t_start >= min_seconds:
            break
    per_layer = float(np.median(times))
    value = batch / (per_layer * layers)
    return {"value": value, "unit": "tokens/s", "cores": NCORES, "kind": "oracle",
            "sample": (f"FP64 numpy oracle (unpack + factored forward) on the 7 linears of one decoder layer, "
                       f"{batch} tokens per call, {len(times)} repetitions ({sum(times):.1f} s), median scaled x{layers} layers; "
                       f"BLAS threads {NCORES}, unpacking single-threaded")}


def run_reference(args, b):
    world, rank, _ = dist_env()
    if rank != 0:
        return
    if args.workload == "prefill":
        ranks7 = [r for (_nm, _m, _n, r) in oracle_shapes()]
    else:
        ranks7 = oracle_ranks(args)[:7]
    data = oracle_layer_sample(b, ranks7)
    for _ in range(max(args.warmup, 0)):
        time_oracle_layer(data)
    times = [time_oracle_layer(data) for _ in range(args.steps)]
    step = float(np.mean(times))
    value = b / (step * args.layers)
    line = {
        "impl": "reference", "metric": METRIC, "value": value, "unit": "tokens/s", "n_gpus": args.gpus,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": step * 1e3,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
        "data": "synthetic (seeded PCG64 signs/scales/activations)",
        "config": config_dict(args),
        "cpu_baseline": {"value": value, "unit": "tokens/s", "cores": NCORES, "kind": "oracle",
                         "sample": (f"each step: FP64 oracle forward of the 7 linears of one decoder layer "
                                    f"(1/{args.layers} of the workload), {b} tokens per call; ms_per_step is "
                                    f"that measured step, value = tokens / (step time x {args.layers} layers)")},
        "e2e": {"value": value, "unit": "tokens/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line))


SCHEDULES = {"dag": "q|k|v and gate|up on parallel streams (decoder dependency DAG)",
             "group": "q|k|v and gate|up each as one multi-layer call (shared input), one stream",
             "serial": "one stream in model order",
             "step": "the whole step as one persistent launch (af1_step_run) in the decoder's level order"}


DECODE_KERNEL_NAMES = {"lut": "lookup tables on the CUDA cores",
                       "mma": "tcgen05 kind::f16 tensor cores (+-b_j FP16 / +-1 BF16 signs)",
                       "tc": "tcgen05 kind::f8f6f4 tensor cores (e4m3 signs and activation terms)"}


def decode_kernel_name(b):
    if DECODE_KERNEL != "auto":
        return DECODE_KERNEL_NAMES[DECODE_KERNEL] + " (layer flag)"
    return DECODE_KERNEL_NAMES[decode_kernel_of(b)] + " (default dispatch)"


def config_dict(args):
    if args.workload == "prefill":
        return {"workload": (f"LLaMA-3-8B-shaped AF1 linears (q,k,v,o,gate,up,down at 1.0-BPW ranks) x {args.layers} "
                             f"layers, prefill {args.tokens} tokens per call, FP16 N(0,1) activations with 1% outlier "
                             f"channels x20, " + SCHEDULES[args.schedule] + ("" if args.no_graph else ", CUDA graph")),
                "tokens": args.tokens, "layers": args.layers, "linears_per_step": 7 * args.layers,
                "l2": "inputs larger than L2 (weights + activations per step >> 129 MB), no flush"}
    if args.ranks == "hisa":
        ranks = ("HiSA-like ranks: each matrix's 1.0-BPW rank x U(0.7, 1.3) (seeded), renormalised to 1.0 BPW over "
                 "the stack")
    else:
        ranks = "1.0-BPW ranks (q,o r2028 / k,v r800 / gate,up,down r3167)"
    return {"workload": (f"LLaMA-3-8B-shaped AF1 decoder linears (q,o 4096x4096 / k,v 1024x4096 / gate,up 14336x4096 "
                         f"/ down 4096x14336), {ranks}, x {args.layers} layers, decode batch {args.batch}, "
                         + SCHEDULES[args.schedule] + ("" if args.no_graph else ", CUDA graph")),
            "batch": args.batch, "layers": args.layers, "linears_per_step": 7 * args.layers, "ranks": args.ranks,
            "stream_layout": ("AF1_MANY_STREAMS (af1_set_stream_layout: the DAG's parallel streams)"
                              if args.schedule == "dag" else "AF1_ONE_STREAM (af1_set_stream_layout)"),
            "decode_kernel": decode_kernel_name(args.batch),
            "l2": "inputs larger than L2 (packed weights per step >> 129 MB), no flush"}


# ---------------------------------------------------------------------------
# Clock sampling during the timed region
# ---------------------------------------------------------------------------

class Clocks:
    Q = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,clocks_event_reasons.hw_slowdown,"
         "clocks_event_reasons.hw_thermal_slowdown,clocks_event_reasons.sw_thermal_slowdown,"
         "clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index):
        self.gpu = gpu_index
        self.proc = None
        self.path = os.path.join("/tmp", f"af1_clocks_{os.getpid()}.csv")

    def start(self):
        try:
            self.f = open(self.path, "w")
            self.proc = subprocess.Popen(["nvidia-smi", "-i", str(self.gpu), f"--query-gpu={self.Q}",
                                          "--format=csv,noheader,nounits", "-lms", "100"],
                                         stdout=self.f, stderr=subprocess.DEVNULL)
        except Exception:
            self.proc = None

    def stop(self):
        if self.proc is None:
            return None
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except Exception:
            self.proc.kill()
        self.f.close()
        sm, mx, reasons = [], 0.0, set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for line in open(self.path):
            parts = [p.strip() for p in line.split(",")]
            if len(parts) < 9:
                continue
            try:
                sm.append(float(parts[1]))
                mx = max(mx, float(parts[2]))
            except ValueError:
                continue
            for nm, v in zip(names, parts[5:9]):
                if v.lower().startswith("active"):
                    reasons.add(nm)
        os.unlink(self.path)
        if not sm:
            return None
        return {"sm_mhz": float(np.median(sm)), "sm_max_mhz": mx, "reasons": sorted(reasons), "samples": len(sm)}


# ---------------------------------------------------------------------------
# The AF1 arm
# ---------------------------------------------------------------------------

def decode_flags():
    """Layer-constructor keywords of the decode kernel chosen on the command line."""
    return {"tc_decode": DECODE_KERNEL == "tc", "mma_decode": DECODE_KERNEL == "mma",
            "lut_decode": DECODE_KERNEL == "lut"}


def build_layers(P, torch, layers, batch, rank, outlier_frac=0.0, ranks=None):
    """7 linears per layer with seeded synthetic words; ranks: one per linear
    (default: every matrix's 1.0-BPW rank)."""
    import synth
    objs = []
    for li in range(layers):
        for si, (name, m, n, r) in enumerate(shapes()):
            if ranks is not None:
                r = ranks[7 * li + si]
            d = synth.layer_words(100000 * (rank + 1) + 7 * li + si, m, n, r, batch, outlier_frac=outlier_frac)
            f16 = lambda bits: torch.from_numpy(np.ascontiguousarray(bits).view(np.float16)).cuda()
            Uw = torch.from_numpy(d["Uw"].view(np.int32)).cuda()
            Vw = torch.from_numpy(d["Vw"].view(np.int32)).cuda()
            layer = P.Layer.from_words(Uw, Vw, f16(d["a"]), f16(d["s"]), f16(d["b"]), m, n, r, **decode_flags(),
                                       any_rank=ranks is not None)
            del Uw, Vw
            x = f16(d["x"]).reshape(batch, n)
            objs.append((name, m, n, r, layer, x))
    return objs


L2_BYTES = 129e6  # GB300 L2; per-shape timings rotate over copies totalling >= 2x this


def device_layer(P, torch, m, n, r, seed, any_rank=False):
    """A layer with seeded random sign words drawn on the device (fast at
    full size; padding bits are cleared by the library's re-layout) and the
    synthetic FP16 scales of synth."""
    import synth
    g = torch.Generator(device="cuda")
    g.manual_seed(seed)
    wu, wv = P.words_per_row(r), P.words_per_row(n)
    Uw = torch.randint(-2**31, 2**31 - 1, (m, wu), generator=g, device="cuda", dtype=torch.int64).to(torch.int32)
    Vw = torch.randint(-2**31, 2**31 - 1, (r, wv), generator=g, device="cuda", dtype=torch.int64).to(torch.int32)
    rs = synth.rng(seed)
    f16 = lambda bits: torch.from_numpy(np.ascontiguousarray(bits).view(np.float16)).cuda()
    a, s_, b = f16(synth.scales_f16(rs, m)), f16(synth.scales_f16(rs, r)), f16(synth.scales_f16(rs, n))
    layer = P.Layer.from_words(Uw, Vw, a, s_, b, m, n, r, any_rank=any_rank, **decode_flags())
    del Uw, Vw
    return layer


def time_graph(torch, fn, stream, reps):
    """ms per call of fn() replayed as a CUDA graph (3 warm-up replays)."""
    with torch.cuda.stream(stream):
        fn()
    torch.cuda.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=stream):
        fn()
    for _ in range(3):
        g.replay()
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    with torch.cuda.stream(stream):
        for _ in range(reps):
            g.replay()
    e1.record(stream)
    torch.cuda.synchronize()
    del g
    return e0.elapsed_time(e1) / reps


def sweep(P, torch, peaks, stream):
    """Per-shape timings: every LLaMA-3-8B shape at 1, 4 and 16 tokens and the
    70B-class shapes at 1 and 8 tokens (decode path, HBM roofline) and at 64
    and 512 tokens (prefill path, tensor roofline); each against dense BF16
    torch.matmul of the same shape. Calls rotate over copies of the layer
    totalling at least twice the L2, so every call streams its weights from
    HBM. Single calls on one stream: the one-stream layout."""
    import math
    import synth
    P.set_stream_layout(P.AF1_ONE_STREAM)
    hbm = peaks.get("hbm_gbs", 6800.0)
    tpk = peaks.get("bf16_tflops_sustained", 1700.0)
    plan = [("q/o", 4096, 4096, (1, 4, 16)), ("k/v", 1024, 4096, (1, 4, 16)),
            ("gate/up", 14336, 4096, (1, 4, 16)), ("down", 4096, 14336, (1, 4, 16))]
    plan += [(f"70b {m}x{n}", m, n, (1, 8, 64, 512)) for (m, n) in synth.LLAMA_70B_SHAPES]
    out = []
    for si, (name, m, n, batches) in enumerate(plan):
        r = P.rank_for_budget(m, n)
        packed = r * (m + n) // 8 + 2 * (m + n + r)
        copies = max(2, min(128, math.ceil(2 * L2_BYTES / packed)))
        layers = [device_layer(P, torch, m, n, r, 7000 + 100 * si + c) for c in range(copies)]
        dense_copies = max(2, math.ceil(2 * L2_BYTES / (2 * m * n)))
        gd = torch.Generator(device="cuda")
        gd.manual_seed(8000 + si)
        dense = [torch.randn((m, n), generator=gd, device="cuda", dtype=torch.bfloat16) * 0.02
                 for _ in range(dense_copies)]
        for b in batches:
            gx = torch.Generator(device="cuda")
            gx.manual_seed(9000 + b)
            x = torch.randn((b, n), generator=gx, device="cuda", dtype=torch.float16)
            y = torch.empty((b, m), device="cuda", dtype=torch.float16)
            ws = torch.zeros(layers[0].workspace_bytes(b), dtype=torch.uint8, device="cuda")

            def run():
                for L in layers:
                    L.forward_into(x, y, ws, stream=stream)
            reps = 5 if b <= 16 else 2
            us = time_graph(torch, run, stream, reps) * 1e3 / copies
            xb = x.to(torch.bfloat16)

            def run_dense():
                for W in dense:
                    torch.matmul(xb, W.t())
            us_dense = time_graph(torch, run_dense, stream, reps) * 1e3 / dense_copies
            e = {"shape": name, "m": m, "n": n, "r": r, "tokens": b, "us_per_call": us,
                 "tokens_per_s": b / (us * 1e-6), "copies": copies, "dense_bf16_us": us_dense,
                 "speedup_vs_dense_bf16": us_dense / us}
            if b <= 16:
                alg = algorithmic_bytes(m, n, r, b)
                e.update({"path": "decode", "kernel": decode_kernel_of(b), "bound": "hbm", "algorithmic_bytes": alg,
                          "achieved_gbs": alg / (us * 1e-6) / 1e9, "frac": alg / (us * 1e-6) / 1e9 / hbm})
            else:
                fl = 2 * b * r * (m + n)
                e.update({"path": "one 16-bit-operand decode pass" if mid_pass_of(m, n, r, b) else "prefill",
                          "bound": "tensor", "flops": fl,
                          "achieved_tflops": fl / (us * 1e-6) / 1e12, "frac": fl / (us * 1e-6) / 1e12 / tpk})
            out.append(e)
            del ws, x, y, xb
        for L in layers:
            L.free()
        del layers, dense
        torch.cuda.empty_cache()
    return out


# The library's default dispatch: passes of more than 4 tokens run on the
# 16-bit-operand tensor-core kernel, passes of 1-4 tokens on the lookup tables.
LUT_MAX_TOKENS = 4


def decode_kernel_of(b):
    """The kernel family the phases of a decode call of b tokens run on, per
    the library's dispatch and the layers' decode-kernel flag."""
    if DECODE_KERNEL != "auto":
        return DECODE_KERNEL
    return "mma" if b > LUT_MAX_TOKENS else "lut"


def mid_pass_of(m, n, r, b):
    """Whether a call of 17..64 tokens runs as one pass of the 16-bit-operand
    decode kernel instead of the prefill kernel (the library's rule: up to 32
    tokens below 70 M signs, up to 64 below 20 M; no LUT or e4m3 flag)."""
    if DECODE_KERNEL in ("lut", "tc") or not 16 < b <= 64:
        return False
    signs = r * (m + n)
    return (b <= 32 and signs <= 70_000_000) or signs <= 20_000_000


def phase_launches(m, n, r, b):
    """Kernel launches of one decode call (b <= 16 tokens): one per phase,
    plus a B-operand preparation launch per phase when the e4m3 tensor-core
    kernel runs a pass of more than 4 tokens."""
    if decode_kernel_of(b) == "tc":
        return 4 if b > 4 else 2
    return 2


def grouped_call(lay, grp, b):
    """A multi-layer call runs as one launch per phase when every phase of
    every layer of the group takes the lookup-table kernel."""
    return decode_kernel_of(b) == "lut"


def step_launches(objs, b, schedule):
    """Kernel launches of one decode step of 7-linear layers."""
    total = 0
    for li in range(len(objs) // 7):
        lay = objs[7 * li:7 * li + 7]
        calls = [phase_launches(m, n, r, b) for (_nm, m, n, r, _L, _x) in lay]
        if schedule == "group":
            for grp in ((0, 1, 2), (4, 5)):
                if grouped_call(lay, grp, b):  # every phase on the lookup-table kernel: one launch per phase
                    total += 2
                else:
                    total += sum(calls[i] for i in grp)
            total += calls[3] + calls[6]
        else:
            total += sum(calls)
    return total


def group_step(P, views, stream, ws, ws_multi):
    """One decode step over views = [(layer, x, y)] * 7 per decoder layer with
    q|k|v and gate|up each as one af1_linear_forward_multi call (the decoder's
    shared inputs), all on one stream."""
    for li in range(len(views) // 7):
        q, k, v, o, gate, up, down = views[7 * li:7 * li + 7]
        P.forward_multi([q[0], k[0], v[0]], q[1], [q[2], k[2], v[2]], ws_multi, stream=stream)
        o[0].forward_into(o[1], o[2], ws, stream=stream)
        P.forward_multi([gate[0], up[0]], gate[1], [gate[2], up[2]], ws_multi, stream=stream)
        down[0].forward_into(down[1], down[2], ws, stream=stream)


def dag_step(torch, views, stream, side, ws, ws_side):
    """One decode step over views = [(layer, x, y)] * 7 per decoder layer on
    the decoder's dependency DAG: per layer q | k | v in parallel, then o, then
    gate | up in parallel, then down (attention and activations are not part
    of this workload). Each parallel branch has its own workspace."""
    for li in range(len(views) // 7):
        q, k, v, o, gate, up, down = views[7 * li:7 * li + 7]
        ev = torch.cuda.Event()
        ev.record(stream)
        for st in side:
            st.wait_event(ev)
        q[0].forward_into(q[1], q[2], ws, stream=stream)
        k[0].forward_into(k[1], k[2], ws_side[0], stream=side[0])
        v[0].forward_into(v[1], v[2], ws_side[1], stream=side[1])
        for st in side:
            e = torch.cuda.Event()
            e.record(st)
            stream.wait_event(e)
        o[0].forward_into(o[1], o[2], ws, stream=stream)
        ev = torch.cuda.Event()
        ev.record(stream)
        side[0].wait_event(ev)
        gate[0].forward_into(gate[1], gate[2], ws, stream=stream)
        up[0].forward_into(up[1], up[2], ws_side[0], stream=side[0])
        e = torch.cuda.Event()
        e.record(side[0])
        stream.wait_event(e)
        down[0].forward_into(down[1], down[2], ws, stream=stream)


def nabf_bench(P, torch):
    """NABF (the factorization that produces the layer) on synthetic
    weights: a rank-512 structure plus noise, LLaMA-3-8B 4096 x 4096 at the
    1.0-BPW rank and a 1024 x 1024 sample, with per-column / per-row
    calibration scales; wall time per iteration on the GPU (the call
    synchronizes), and the FP64 oracle on the host for the small sample."""
    import time
    import synth
    out = {"workload": "NABF on synthetic W (rank-512 structure + N(0, 0.01) noise, i, o ~ U(0.5, 2)), "
                       "rho 1e-2, eta 0.01, 20 power iterations; wall time per iteration (iterations 1..5 "
                       "minus the initialization)"}
    for (m, n) in ((1024, 1024), (4096, 4096)):
        r = P.rank_for_budget(m, n)
        g = synth.rng(m)
        k = min(512, r // 2)
        W = (g.normal(size=(m, k)) @ g.normal(size=(k, n)) * 0.01 + g.normal(0.0, 0.01, size=(m, n))).astype(np.float32)
        i_s, o_s = g.uniform(0.5, 2.0, n).astype(np.float32), g.uniform(0.5, 2.0, m).astype(np.float32)
        Wt, it, ot = (torch.from_numpy(v).cuda() for v in (W, i_s, o_s))
        times = {}
        for iters in (0, 5):
            P.nabf_factorize(Wt, r, iters=iters, rho=1e-2, in_scale=it, out_scale=ot)  # warm-up (library loads)
            t0 = time.perf_counter()
            res = P.nabf_factorize(Wt, r, iters=iters, rho=1e-2, in_scale=it, out_scale=ot)
            times[iters] = time.perf_counter() - t0
        row = {"m": m, "n": n, "r": r, "gpu_ms_per_iteration": (times[5] - times[0]) / 5 * 1e3,
               "gpu_init_ms": times[0] * 1e3, "objective": res["objective"], "q_left": res["q_left"],
               "q_right": res["q_right"]}
        if m == 1024:
            from oracle import af1_nabf_oracle as N
            t0 = time.perf_counter()
            N.nabf(W, r, 0, rho=1e-2, in_scale=i_s, out_scale=o_s)
            t1 = time.perf_counter()
            ref = N.nabf(W, r, 2, rho=1e-2, in_scale=i_s, out_scale=o_s)
            t2 = time.perf_counter()
            row["cpu_oracle_s_per_iteration"] = ((t2 - t1) - (t1 - t0)) / 2
            row["cpu_oracle_objective_2_iters"] = list(ref["objective"])
        out[f"{m}x{n}"] = row
    return out


def mlp_swiglu(P, torch, stream, steps):
    """LLaMA-3-8B MLP blocks at one token: gate | up (parallel streams), then
    the down projection of h = FP16(SiLU(gate) * up). Fused: the down call
    forms h itself (af1_linear_forward_swiglu); unfused: h by torch
    elementwise ops, then af1_linear_forward. 32 blocks rotate (weights far
    larger than L2); CUDA graph; the many-streams layout (two streams)."""
    P.set_stream_layout(P.AF1_MANY_STREAMS)
    blocks = 32
    rank = P.rank_for_budget
    mk = lambda m, n, seed: device_layer(P, torch, m, n, rank(m, n), seed)
    gates = [mk(14336, 4096, 5000 + 3 * i) for i in range(blocks)]
    ups = [mk(14336, 4096, 5001 + 3 * i) for i in range(blocks)]
    downs = [mk(4096, 14336, 5002 + 3 * i) for i in range(blocks)]
    g = torch.Generator(device="cuda")
    g.manual_seed(77)
    x = torch.randn((1, 4096), generator=g, device="cuda", dtype=torch.float16)
    gy = torch.empty((1, 14336), device="cuda", dtype=torch.float16)
    uy = torch.empty_like(gy)
    h = torch.empty_like(gy)
    y = torch.empty((1, 4096), device="cuda", dtype=torch.float16)
    nbytes = max(downs[0].workspace_bytes_swiglu(1), gates[0].workspace_bytes(1))
    ws = torch.zeros(nbytes, dtype=torch.uint8, device="cuda")
    ws_side = torch.zeros_like(ws)
    side = torch.cuda.Stream()

    def run(fused):
        for i in range(blocks):
            ev = torch.cuda.Event()
            ev.record(stream)
            side.wait_event(ev)
            gates[i].forward_into(x, gy, ws, stream=stream)
            ups[i].forward_into(x, uy, ws_side, stream=side)
            e = torch.cuda.Event()
            e.record(side)
            stream.wait_event(e)
            if fused:
                downs[i].forward_swiglu_into(gy, uy, y, ws, stream=stream)
            else:
                with torch.cuda.stream(stream):
                    h.copy_(torch.nn.functional.silu(gy.float()).mul_(uy.float()))
                downs[i].forward_into(h, y, ws, stream=stream)

    reps = max(2, steps // 10)
    fused_us = time_graph(torch, lambda: run(True), stream, reps) * 1e3 / blocks
    unfused_us = time_graph(torch, lambda: run(False), stream, reps) * 1e3 / blocks
    for L in gates + ups + downs:
        L.free()
    return {"workload": "32 LLaMA-3-8B MLP blocks, 1 token: gate | up on two streams, then down on "
                        "h = FP16(SiLU(gate) * up); CUDA graph",
            "fused_us_per_block": fused_us, "unfused_us_per_block": unfused_us,
            "unfused": "h by torch elementwise ops (FP32 SiLU and product, FP16 store), then af1_linear_forward"}


def stream_layout_for(P, schedule):
    """AF1_MANY_STREAMS for the decoder DAG (parallel streams), AF1_ONE_STREAM
    for the one-stream schedules."""
    return P.AF1_MANY_STREAMS if schedule == "dag" else P.AF1_ONE_STREAM


def stack_other_ranks(P, torch, peaks, stream, steps, args):
    """The 32-layer stack with the other rank allocation than the headline's
    (uniform 1.0-BPW ranks when the headline uses HiSA-like ranks, and vice
    versa), one token, on the decoder DAG, CUDA graph; weights drawn on the
    device."""
    import synth
    other = "uniform" if args.ranks == "hisa" else "hisa"
    mn = [(m, n) for _ in range(LAYERS) for (_nm, m, n) in synth.LLAMA3_8B_LINEARS]
    ranks = hisa_ranks(mn) if other == "hisa" else [P.rank_for_budget(m, n) for (m, n) in mn]
    layers = [device_layer(P, torch, m, n, r, 20000 + i, any_rank=True) for i, ((m, n), r) in enumerate(zip(mn, ranks))]
    gx = torch.Generator(device="cuda")
    gx.manual_seed(31)
    xs = [torch.randn((1, n), generator=gx, device="cuda", dtype=torch.float16) for (m, n) in mn]
    ys = [torch.empty((1, m), device="cuda", dtype=torch.float16) for (m, n) in mn]
    ws = torch.zeros(max(L.workspace_bytes(1) for L in layers), dtype=torch.uint8, device="cuda")
    side = [torch.cuda.Stream(), torch.cuda.Stream()]
    ws_side = [torch.zeros_like(ws), torch.zeros_like(ws)]
    views = list(zip(layers, xs, ys))
    group = args.schedule == "group"
    if group:
        ws_multi = torch.zeros(max(max(P.workspace_bytes_multi([layers[7 * li + j] for j in (0, 1, 2)], 1),
                                       P.workspace_bytes_multi([layers[7 * li + j] for j in (4, 5)], 1))
                                   for li in range(LAYERS)), dtype=torch.uint8, device="cuda")

        def run():
            group_step(P, views, stream, ws, ws_multi)
    else:
        def run():
            dag_step(torch, views, stream, side, ws, ws_side)
    P.set_stream_layout(stream_layout_for(P, args.schedule))
    ms_dag = time_graph(torch, run, stream, max(5, min(steps, 20)))
    alg = sum(algorithmic_bytes(m, n, r, 1) for (m, n), r in zip(mn, ranks))
    bits = sum(P.storage_bits(m, n, r) for (m, n), r in zip(mn, ranks))
    out = {"workload": f"32 x 7 LLaMA-3-8B linears, {other} ranks, 1 token, "
                       f"{'q|k|v and gate|up as grouped calls, one stream' if group else 'decoder DAG'}, CUDA graph",
           "ranks": other, "ms_per_token": ms_dag, "tokens_per_s": 1e3 / ms_dag,
           "us_per_linear": ms_dag * 1e3 / len(mn), "bpw": bits / sum(m * n for (m, n) in mn),
           "rank_min": min(ranks), "rank_max": max(ranks), "achieved_gbs": alg / (ms_dag * 1e-3) / 1e9,
           "frac": alg / (ms_dag * 1e-3) / 1e9 / peaks.get("hbm_gbs", 6800.0)}
    for L in layers:
        L.free()
    del layers, xs, ys, ws, ws_side, views
    torch.cuda.empty_cache()
    return out


def chained_views(objs, b, dev, torch):
    """The stack's linears reading each other's outputs as a decoder does:
    q, k, v read the layer input, o reads q, gate and up read o, down reads
    h = FP16(SiLU(gate) up), the next layer reads down (the first layer's input
    is an external buffer). Returns (linear, x, y, level[, x2]) items."""
    items = []
    x = objs[0][5]
    for li in range(len(objs) // 7):
        lay = objs[7 * li:7 * li + 7]
        yv = [torch.empty((b, m), dtype=torch.float16, device=dev) for (_n, m, n, r, L, xx) in lay]
        base = 4 * li
        items += [(lay[0][4], x, yv[0], base), (lay[1][4], x, yv[1], base), (lay[2][4], x, yv[2], base),
                  (lay[3][4], yv[0], yv[3], base + 1), (lay[4][4], yv[3], yv[4], base + 2),
                  (lay[5][4], yv[3], yv[5], base + 2), (lay[6][4], yv[4], yv[6], base + 3, yv[5])]
        x = yv[6]
    return items


def prefill_extra(P, torch, peaks, stream, steps):
    """Config 2 inside the default run: the seven LLaMA-3-8B linears at their
    1.0-BPW ranks over 4 layers, 2048 tokens per call (FP16 N(0, 1) with a
    seeded 1 % of channels x20), the tensor-core prefill kernels on the
    decoder DAG, CUDA graph."""
    T, nl = 2048, 4
    objs = build_layers(P, torch, nl, T, 7, outlier_frac=0.01)
    ys = [torch.empty((T, m), dtype=torch.float16, device="cuda") for (_n, m, n, r, L, x) in objs]
    ws = torch.zeros(max(o[4].workspace_bytes(T) for o in objs), dtype=torch.uint8, device="cuda")
    side = [torch.cuda.Stream(), torch.cuda.Stream()]
    ws_side = [torch.zeros_like(ws), torch.zeros_like(ws)]
    views = [(o[4], o[5], y) for o, y in zip(objs, ys)]
    ms = time_graph(torch, lambda: dag_step(torch, views, stream, side, ws, ws_side), stream, max(5, min(steps, 20)))
    P.workspace_status(ws)
    flops = sum(2 * T * r * (m + n) for (_n, m, n, r, L, x) in objs)
    tflops = flops / (ms * 1e-3) / 1e12
    tpeak = peaks.get("bf16_tflops_sustained", 1700.0)
    out = {"workload": "config 2: LLaMA-3-8B linears (1.0-BPW ranks) x 4 layers, 2048 tokens per call, FP16 N(0,1) "
                       "activations with 1% outlier channels x20, decoder DAG, CUDA graph",
           "ms_per_step": ms, "tokens_per_s": T / (ms * 1e-3),
           "roofline": {"bound": "tensor", "kernel": "prefill_kernel (tcgen05 kind::f16, two GEMMs per call)",
                        "achieved": tflops, "peak": tpeak, "unit": "TFLOP/s", "frac": tflops / tpeak,
                        "peak_source": "MEASURED_PEAKS.json bf16_tflops_sustained (FP16 dense rate = BF16 rate)",
                        "algorithmic_flops_per_step": flops}}
    for (_n, m, n, r, L, x) in objs:
        L.free()
    del objs, ys, ws, ws_side, views
    torch.cuda.empty_cache()
    return out


def main():
    global DECODE_KERNEL
    args = parse()
    DECODE_KERNEL = "tc" if args.tc_decode else args.decode_kernel
    b = resolve_workload(args)
    if args.impl == "reference":
        run_reference(args, b)
        return
    import torch
    import torch.distributed as dist

    world, rank, local = dist_env()
    if world > 1:
        torch.cuda.set_device(local)
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
    else:
        torch.cuda.set_device(0)
    import paper_2609_06161_gb300 as P

    if args.shape:
        run_shape(P, torch, args, b)
        return
    dev = torch.device("cuda", torch.cuda.current_device())
    ranks = workload_ranks(args)
    objs = build_layers(P, torch, args.layers, b, rank, outlier_frac=0.01 if args.workload == "prefill" else 0.0,
                        ranks=ranks if args.workload == "decode" else None)
    ws = torch.zeros(max(o[4].workspace_bytes(b) for o in objs), dtype=torch.uint8, device=dev)
    # Inputs and outputs live in one device buffer each so the e2e leg can move
    # them with a single copy per direction.
    xs = [o[5] for o in objs]
    xoff, yoff, xo, yo = [], [], 0, 0
    for (name, m, n, r, layer, x) in objs:
        xoff.append(xo)
        xo += b * n
        yoff.append(yo)
        yo += b * m
    xbuf = torch.empty(xo, dtype=torch.float16, device=dev)
    ybuf = torch.empty(yo, dtype=torch.float16, device=dev)
    for i, x in enumerate(xs):
        xbuf[xoff[i]:xoff[i] + x.numel()].copy_(x.reshape(-1))
    views = []
    for i, (name, m, n, r, layer, x) in enumerate(objs):
        views.append((layer, xbuf[xoff[i]:xoff[i] + b * n].view(b, n), ybuf[yoff[i]:yoff[i] + b * m].view(b, m)))

    stream = torch.cuda.Stream()
    side = [torch.cuda.Stream(), torch.cuda.Stream()]
    ws_side = [torch.zeros_like(ws), torch.zeros_like(ws)]

    def step_serial():
        for (layer, xv, yv) in views:
            layer.forward_into(xv, yv, ws, stream=stream)

    def step_dag():
        dag_step(torch, views, stream, side, ws, ws_side)

    ws_multi = None
    if len(views) % 7 == 0:
        nbytes = max(max(P.workspace_bytes_multi([views[7 * li + j][0] for j in (0, 1, 2)], b),
                         P.workspace_bytes_multi([views[7 * li + j][0] for j in (4, 5)], b))
                     for li in range(len(views) // 7))
        ws_multi = torch.zeros(nbytes, dtype=torch.uint8, device=dev)

    def step_group():
        # q, k, v read one input and gate, up another (the decoder's shared
        # activations): one multi-layer call each.
        group_step(P, views, stream, ws, ws_multi)

    def make_graph(fn, name):
        # The library's stream layout suits the schedule: several streams for
        # the DAG, one stream otherwise (af1_set_stream_layout).
        P.set_stream_layout(stream_layout_for(P, name))
        with torch.cuda.stream(stream):
            fn()
        torch.cuda.synchronize()
        if args.no_graph:
            class _Eager:
                def replay(self):
                    with torch.cuda.stream(stream):
                        fn()
            return _Eager()
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=stream):
            fn()
        torch.cuda.synchronize()
        return g

    # The whole step as one persistent launch, in the DAG's level order.
    step_plan = None
    if len(views) % 7 == 0 and b <= 4 and args.workload == "decode":
        lv7 = [0, 0, 0, 1, 2, 2, 3]
        step_plan = P.Step([(L, xv, yv, 4 * (i // 7) + lv7[i % 7]) for i, (L, xv, yv) in enumerate(views)])
        ws_step = step_plan.make_workspace(dev)

    def step_one_launch():
        step_plan.run(ws_step, stream=stream)

    steps_by_name = {"dag": step_dag, "group": step_group, "serial": step_serial}
    if step_plan is not None:
        steps_by_name["step"] = step_one_launch
    if args.schedule == "step" and step_plan is None:
        raise SystemExit("--schedule step needs the 7-linear decode workload with at most 4 tokens")
    step_name = args.schedule if len(views) % 7 == 0 else "serial"
    graph = make_graph(steps_by_name[step_name], step_name)

    def barrier():
        if world > 1:
            dist.barrier()
        torch.cuda.synchronize()

    for _ in range(max(args.warmup, 3)):
        graph.replay()
    barrier()
    clocks = Clocks(local)
    clocks.start()
    time.sleep(0.3)
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    barrier()
    e0.record(stream)
    with torch.cuda.stream(stream):
        for _ in range(args.steps):
            graph.replay()
    e1.record(stream)
    barrier()
    ms = e0.elapsed_time(e1)
    clk = clocks.stop()
    ms_max = max_over_ranks(dist, torch, world, ms, dev)
    ms_step = ms_max / args.steps
    value = job_tokens_per_s(b, world, args.steps, ms_max * 1e-3)
    nlin = len(views)
    us_layer = ms_step * 1e3 / nlin
    alg = sum(algorithmic_bytes(m, n, r, b) for (name, m, n, r, layer, x) in objs)
    achieved_gbs = alg / (ms_step * 1e-3) / 1e9

    # The same step on the other schedules (outside the headline's timing).
    others = {}
    if len(views) % 7 == 0 and args.workload == "decode":
        for name, fn in steps_by_name.items():
            if name == args.schedule:
                continue
            g2 = make_graph(fn, name)
            for _ in range(3):
                g2.replay()
            torch.cuda.synchronize()
            f0, f1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            f0.record(stream)
            with torch.cuda.stream(stream):
                for _ in range(args.steps):
                    g2.replay()
            f1.record(stream)
            torch.cuda.synchronize()
            sms = f0.elapsed_time(f1) / args.steps
            others[name] = {"ms_per_step": sms, "us_per_layer": sms * 1e3 / len(views), "tokens_per_s": b / (sms * 1e-3)}
            del g2
        if step_plan is not None:
            # The one-launch step with the decoder's data flow: each linear
            # reads its producer's output (the same weights and level order).
            chained = P.Step(chained_views(objs, b, dev, torch))
            ws_ch = chained.make_workspace(dev)
            with torch.cuda.stream(stream):
                for _ in range(3):
                    chained.run(ws_ch, stream=stream)
            torch.cuda.synchronize()
            f0, f1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            f0.record(stream)
            for _ in range(args.steps):
                chained.run(ws_ch, stream=stream)
            f1.record(stream)
            torch.cuda.synchronize()
            P.workspace_status(ws_ch, stream)
            sms = f0.elapsed_time(f1) / args.steps
            others["step_chained"] = {"ms_per_step": sms, "us_per_layer": sms * 1e3 / len(views),
                                      "tokens_per_s": b / (sms * 1e-3),
                                      "inputs": "q,k,v <- layer input, o <- q, gate,up <- o, down <- SwiGLU(gate, up), "
                                                "next layer <- down"}
            chained.destroy()
            del ws_ch
    serial = others.get("serial")

    # e2e: host buffers in pinned memory, copies inside the timed region.
    xh = torch.empty(xo, dtype=torch.float16, pin_memory=True)
    xh.copy_(xbuf.cpu())
    yh = torch.empty(yo, dtype=torch.float16, pin_memory=True)
    for _ in range(3):
        with torch.cuda.stream(stream):
            xbuf.copy_(xh, non_blocking=True)
            graph.replay()
            yh.copy_(ybuf, non_blocking=True)
        stream.synchronize()
    barrier()
    t0 = time.perf_counter()
    for _ in range(args.steps):
        with torch.cuda.stream(stream):
            xbuf.copy_(xh, non_blocking=True)
            graph.replay()
            yh.copy_(ybuf, non_blocking=True)
        stream.synchronize()
    e2e_s = time.perf_counter() - t0
    e2e_value = job_tokens_per_s(b, world, args.steps, max_over_ranks(dist, torch, world, e2e_s, dev))

    dense = None
    if not args.no_dense and rank == 0:
        dense = dense_bf16(torch, objs, b, args, stream)
    peaks = load_peaks()
    sweep_rows = stack = mlp = nabf = prefill = None
    if args.workload == "decode" and rank == 0:
        # Extra measurements, outside the timed region of the headline number.
        if step_plan is not None:
            step_plan.destroy()
            step_plan = None
        if not args.no_stack:
            stack = stack_other_ranks(P, torch, peaks, stream, args.steps, args)
            mlp = mlp_swiglu(P, torch, stream, args.steps)
            nabf = nabf_bench(P, torch)
            prefill = prefill_extra(P, torch, peaks, stream, args.steps)
        if not args.no_sweep:
            sweep_rows = sweep(P, torch, peaks, stream)

    if rank == 0:
        hbm = peaks.get("hbm_gbs")
        if args.workload == "prefill":
            flops = sum(2 * b * r * (m + n) for (name, m, n, r, layer, x) in objs)
            tflops = flops / (ms_step * 1e-3) / 1e12
            tpeak = peaks.get("bf16_tflops_sustained", 1700.0)
            roof = {"bound": "tensor", "kernel": "af1_linear_forward prefill (two tcgen05 kind::f16 GEMM kernels per call)",
                    "achieved": tflops, "peak": tpeak, "unit": "TFLOP/s", "frac": tflops / tpeak,
                    "peak_source": "MEASURED_PEAKS.json bf16_tflops_sustained (FP16 dense rate = BF16 rate)",
                    "algorithmic_flops_per_step": flops, "traffic": None}
        else:
            # DRAM bytes (read + write) of one layer's 14 lookup-table kernels
            # at one token, from the ncu capture summarised in
            # profiles/lut_kernel_llama3_8b_b1.md, times 32 layers.
            traffic = None
            if b == 1 and decode_kernel_of(b) == "lut" and args.schedule == "dag":
                traffic = (DECODE_TRAFFIC_B1_PER_LAYER * args.layers if args.ranks == "uniform"
                           else int(round(DECODE_TRAFFIC_RATIO_HISA_B1 * alg)))
            elif (b == 1 and decode_kernel_of(b) == "lut" and args.schedule == "group" and args.ranks == "hisa"
                  and DECODE_TRAFFIC_RATIO_HISA_B1_GROUP is not None):
                traffic = int(round(DECODE_TRAFFIC_RATIO_HISA_B1_GROUP * alg))
            fam = decode_kernel_of(b)
            kname = ("af1_step_run (one persistent step_kernel launch per step)" if args.schedule == "step" else
                     "af1_linear_forward (two 16-bit-operand tensor-core kernels per call, hdecode_kernel<1|2>)"
                     if fam == "mma" else
                     "af1_linear_forward (two e4m3 tensor-core kernels per call, decode_kernel<1|2>, with "
                     "bprep_kernel for passes of more than 4 tokens)" if fam == "tc" else
                     "af1_linear_forward_multi / af1_linear_forward (two lookup-table kernels per call, "
                     "lut_kernel<1|2>)" if args.schedule == "group" else
                     "af1_linear_forward (two lookup-table kernels per call, lut_kernel<1|2>, stream_kernel<1|2> "
                     "for the largest matrices)")
            roof = {"bound": "hbm", "kernel": kname,
                    "achieved": achieved_gbs, "peak": hbm, "unit": "GB/s",
                    "frac": (achieved_gbs / hbm) if hbm else None, "peak_source": "MEASURED_PEAKS.json hbm_gbs"
                    if "hbm_gbs" in peaks else "fallback 6800 GB/s",
                    "algorithmic_bytes_per_step": alg, "traffic": traffic,
                    "traffic_source": ("ncu dram__bytes_read.sum + dram__bytes_write.sum of the step's lookup-table "
                                       "launches, captured on a smaller stack of the same workload and scaled "
                                       "(uniform: per layer x layers; HiSA: by algorithmic bytes)") if traffic else None}
        line = {
            "metric": METRIC, "value": value, "unit": "tokens/s", "n_gpus": world, "steps": args.steps,
            "warmup": max(args.warmup, 3), "ms_per_step": ms_step, "us_per_layer": us_layer,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
            "dtype": "f16" if args.workload == "prefill" else "f32",
            "data": "synthetic (seeded PCG64 packed signs, |N(0,0.02)|+1e-3 scales, N(0,1) activations)",
            "config": config_dict(args),
            "roofline": roof,
            "e2e": {"value": e2e_value, "unit": "tokens/s", "h2d_bytes_per_step": xo * 2,
                    "d2h_bytes_per_step": yo * 2},
            "gpu_launches": ((1 if args.schedule == "step" else step_launches(objs, b, args.schedule))
                             if args.workload == "decode" and nlin % 7 == 0 else 2 * nlin) * args.steps,
            "clocks": clk,
        }
        if dense is not None:
            line["dense_bf16_baseline"] = dense
        if serial is not None:
            line["serial_chain"] = serial
        if others:
            line["other_schedules"] = others
        if stack is not None:
            line["stack_other_ranks"] = stack
        if prefill is not None:
            line["prefill"] = prefill
        if mlp is not None:
            line["mlp_swiglu"] = mlp
        if nabf is not None:
            line["nabf"] = nabf
        if sweep_rows is not None:
            line["sweep"] = sweep_rows
        if not args.no_cpu and world == 1 and args.workload == "decode":
            line["cpu_baseline"] = cpu_baseline(b, args.layers, oracle_ranks(args)[:7])
        if args.workload == "prefill":
            line["dtype"] = "f16 tcgen05 MMA / f32 accumulate (1-bit signs expanded to +-b, f16 activations)"
            line["us_per_layer"] = ms_step * 1e3 / nlin
        print(json.dumps(line))
    if world > 1:
        dist.destroy_process_group()


def run_shape(P, torch, args, b):
    """One linear of shape --shape at its 1.0-BPW rank and b tokens (--batch,
    or --tokens with --workload prefill):
    --warmup then --steps calls, each on the next of enough copies of the
    layer to exceed twice the L2 (every call streams its signs from HBM), in
    a CUDA graph or (--no-graph) as eager launches for profilers."""
    import math
    m, n = (int(v) for v in args.shape.lower().split("x"))
    r = P.rank_for_budget(m, n)
    packed = r * (m + n) // 8 + 2 * (m + n + r)
    copies = max(2, min(128, math.ceil(2 * L2_BYTES / packed)))
    layers = [device_layer(P, torch, m, n, r, 7000 + c) for c in range(copies)]
    g = torch.Generator(device="cuda")
    g.manual_seed(9000 + b)
    x = torch.randn((b, n), generator=g, device="cuda", dtype=torch.float16)
    y = torch.empty((b, m), device="cuda", dtype=torch.float16)
    ws = torch.zeros(layers[0].workspace_bytes(b), dtype=torch.uint8, device="cuda")
    stream = torch.cuda.Stream()
    calls = max(args.steps, 1)

    def run(k):
        for i in range(k):
            layers[i % copies].forward_into(x, y, ws, stream=stream)

    if args.no_graph:
        with torch.cuda.stream(stream):
            run(max(args.warmup, 1))
        torch.cuda.synchronize()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        with torch.cuda.stream(stream):
            run(calls)
        e1.record(stream)
        torch.cuda.synchronize()
        us = e0.elapsed_time(e1) * 1e3 / calls
    else:
        us = time_graph(torch, lambda: run(copies), stream, max(1, calls // copies)) * 1e3 / copies
    P.workspace_status(ws)
    peaks = load_peaks()
    alg = algorithmic_bytes(m, n, r, b)
    fl = 2 * b * r * (m + n)
    line = {"shape": f"{m}x{n}", "rank": r, "tokens": b, "us_per_call": us, "copies": copies,
            "graph": not args.no_graph, "algorithmic_bytes": alg, "achieved_gbs": alg / (us * 1e-6) / 1e9,
            "hbm_frac": alg / (us * 1e-6) / 1e9 / peaks.get("hbm_gbs", 6800.0),
            "flops": fl, "achieved_tflops": fl / (us * 1e-6) / 1e12,
            "tensor_frac": fl / (us * 1e-6) / 1e12 / peaks.get("bf16_tflops_sustained", 1700.0)}
    print(json.dumps(line))
    for L in layers:
        L.free()


def load_peaks():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            return json.load(f)
    except Exception:
        return {"hbm_gbs": 6800.0}


def dense_bf16(torch, objs, b, args, stream):
    """Same step with dense BF16 weights and torch.matmul (cuBLAS): a reported
    baseline, not part of the AF1 path."""
    g = torch.Generator(device="cuda")
    g.manual_seed(1234)
    ws, xs = [], []
    for (name, m, n, r, layer, x) in objs:
        ws.append(torch.randn((m, n), generator=g, device="cuda", dtype=torch.bfloat16) * 0.02)
        xs.append(x.to(torch.bfloat16))
    ys = [None] * len(ws)

    def step():
        for i in range(len(ws)):
            ys[i] = torch.matmul(xs[i], ws[i].t())

    with torch.cuda.stream(stream):
        step()
    torch.cuda.synchronize()
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph, stream=stream):
        step()
    for _ in range(3):
        graph.replay()
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    steps = max(5, min(args.steps, 20))
    e0.record(stream)
    with torch.cuda.stream(stream):
        for _ in range(steps):
            graph.replay()
    e1.record(stream)
    torch.cuda.synchronize()
    ms = e0.elapsed_time(e1) / steps
    nbytes = sum(w.numel() * 2 for w in ws)
    del ws, xs, ys, graph
    torch.cuda.empty_cache()
    return {"ms_per_step": ms, "tokens_per_s": b / (ms * 1e-3), "weight_bytes": nbytes,
            "achieved_gbs": nbytes / (ms * 1e-3) / 1e9}


if __name__ == "__main__":
    main()
