"""Launch plans of the 16-bit-operand tensor-core decode kernel, checked on the
CPU (af1_mma_plan_dry: the planner the launcher calls, run on the host).

Every plan must fit what the kernel assumes: B rows for all the pass's
tokens (two BF16 terms of s' per token in phase 2 up to 16 tokens, one FP16
term in one-pass calls of 17-64), the CTA's 256 tensor-memory columns for
its accumulators and A ring, at most two CTAs per SM (so two CTAs' tensor
memory always fits the SM's 512 columns), clusters of 1-16 CTAs that cover
every 128-column chunk with at least one chunk each, and the device's
shared memory. Shapes: every LLaMA-3-8B and 70B-class matrix of the
workloads at its 1.0-BPW rank, ragged shapes, and the longest contraction.
"""
import os
import subprocess
import sys

import pytest

from oracle import af1_oracle as O

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
SMS, MAX_SMEM = 152, 232448  # GB300: SMs, opt-in shared memory per block
SM_SMEM = 233472             # shared memory per SM


def _lib():
    so = os.path.join(ROOT, "paper_2609_06161_gb300", "libaf1.so")
    if not os.path.exists(so):
        subprocess.run([sys.executable, os.path.join(ROOT, "paper_2609_06161_gb300", "build.py")], check=True)
    import paper_2609_06161_gb300 as P
    return P


def _matrices():
    shapes = [(4096, 4096), (1024, 4096), (14336, 4096), (4096, 14336),
              (8192, 8192), (1024, 8192), (28672, 8192), (8192, 28672)]
    out = []
    for (m, n) in shapes:
        r = O.rank_for_budget(m, n, 1)
        out += [(r, n), (m, r)]  # phase 1 (B = V^T), phase 2 (U)
    out += [(77, 130), (100, 77), (321, 700), (1000, 321), (100, 1920), (2028, 32768), (256, 2028), (5, 9)]
    return sorted(set(out))


def _check(P, phase, R, C, T):
    p = P.mma_plan_dry(phase, R, C, T, SMS, MAX_SMEM)
    if not p["ok"]:
        return p
    terms = 1 if phase == 1 else (2 if T <= 16 else 1)
    assert p["rows"] in (16, 32, 64) and p["rows"] >= terms * T, p
    assert p["accumulators"] >= 1 and p["ring"] >= 1, p
    assert p["tmem_cols"] == p["accumulators"] * p["rows"] + 64 * p["ring"] <= 256, p
    nch = -(-C // 128)
    assert 1 <= p["ks"] <= 16 and 1 <= p["cpc"] <= 64, p
    assert (p["ks"] - 1) * p["cpc"] < nch <= p["ks"] * p["cpc"], p  # every CTA has a chunk, every chunk a CTA
    assert p["smem"] <= MAX_SMEM, p
    assert SM_SMEM // p["smem"] <= 2, p  # at most two CTAs (512 tensor-memory columns) per SM
    assert p["grid_x"] == -(-R // 128) and p["grid_y"] == p["ks"], p
    return p


@pytest.mark.parametrize("tokens", [1, 4, 5, 8, 9, 12, 16])
def test_decode_plans_fit(tokens):
    P = _lib()
    for (R, C) in _matrices():
        for phase in (1, 2):
            p = _check(P, phase, R, C, tokens)
            # every workload matrix has a plan at every decode width
            if C <= 28672:
                assert p["ok"], (phase, R, C, tokens)


@pytest.mark.parametrize("tokens", [17, 24, 32, 33, 48, 64])
def test_one_pass_plans_fit(tokens):
    P = _lib()
    for (R, C) in _matrices():
        for phase in (1, 2):
            p = _check(P, phase, R, C, tokens)
            # the small layers the one-pass rule takes (below 20 M signs) have plans
            if R * C <= 10_000_000 and C <= 8192:
                assert p["ok"], (phase, R, C, tokens)


def test_plan_query_rejects_bad_arguments():
    P = _lib()
    for args in ((3, 100, 100, 4), (1, 0, 100, 4), (1, 100, 40000, 4), (1, 100, 100, 0), (2, 100, 100, 65)):
        with pytest.raises(P.AF1Error) as e:
            P.mma_plan_dry(*args)
        assert e.value.code == -1
