"""The C ABI library: it loads, exports every entry point include/af1.h
declares, and its host-only logic (rank rule, argument validation that needs
no device) behaves as documented. No GPU compute is called here."""
import ctypes
import os
import re
import subprocess
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
LIB = os.path.join(ROOT, "paper_2609_06161_gb300", "libaf1.so")


def _ensure_built():
    if not os.path.exists(LIB):
        subprocess.run([sys.executable, os.path.join(ROOT, "paper_2609_06161_gb300", "build.py")], check=True)


def declared_functions():
    src = open(os.path.join(ROOT, "include", "af1.h")).read()
    return sorted(set(re.findall(r"AF1_API\s+[\w\s\*]*?\b(af1_\w+)\s*\(", src)))


def test_header_declares_the_boundary():
    names = declared_functions()
    for required in ("af1_pack_layer", "af1_linear_forward", "af1_free", "af1_last_error"):
        assert required in names


def test_library_exports_every_declared_symbol():
    _ensure_built()
    out = subprocess.run(["nm", "-D", "--defined-only", LIB], capture_output=True, text=True, check=True).stdout
    exported = {line.split()[-1] for line in out.splitlines() if " T " in line}
    missing = [f for f in declared_functions() if f not in exported]
    assert not missing, missing
    lib = ctypes.CDLL(LIB)
    for f in declared_functions():
        getattr(lib, f)


def test_rank_rule_matches_oracle():
    _ensure_built()
    import paper_2609_06161_gb300 as P
    from oracle import af1_oracle as O
    from fractions import Fraction
    shapes = [(4096, 4096), (1024, 4096), (14336, 4096), (4096, 14336), (8192, 8192), (1024, 8192),
              (28672, 8192), (8192, 28672), (7, 9), (4, 4), (100, 33), (1, 1000)]
    for (m, n) in shapes:
        for num, den in ((1, 1), (5, 2), (1, 2), (3, 1)):
            assert P.rank_for_budget(m, n, num, den) == O.rank_for_budget(m, n, Fraction(num, den)), (m, n, num, den)


def test_storage_bits_matches_oracle():
    _ensure_built()
    import paper_2609_06161_gb300 as P
    from oracle import af1_oracle as O
    for (m, n, r) in [(4096, 4096, 2028), (1024, 4096, 800), (28672, 8192, 6352), (7, 9, 3), (1, 1, 1)]:
        assert P.storage_bits(m, n, r) == O.storage_bits(m, n, r), (m, n, r)
    with pytest.raises(P.AF1Error):
        P.storage_bits(4, 4, 0)


def test_hisa_allocation_respects_budget():
    # bench.hisa_ranks: +-30 % draws renormalised so that the stack stays at
    # (not above) 1.0 BPW, with less than one rank step of slack.
    _ensure_built()
    import bench
    from oracle import af1_oracle as O
    import synth
    shapes = [(m, n) for (_nm, m, n) in synth.LLAMA3_8B_LINEARS] * 4
    ranks = bench.hisa_ranks(shapes, seed=3)
    mats = [(m, n, r) for (m, n), r in zip(shapes, ranks)]
    budget = sum(m * n for (m, n) in shapes)
    total = sum(O.storage_bits(m, n, r) for (m, n, r) in mats)
    assert total <= budget
    assert all(total + (m + n + 16) > budget for (m, n, _r) in mats)
    base = [O.rank_for_budget(m, n, 1) for (m, n) in shapes]
    assert any(r != b for r, b in zip(ranks, base))
    assert all(0.6 * b <= r <= 1.4 * b for r, b in zip(ranks, base))


def test_host_validation_errors():
    _ensure_built()
    import paper_2609_06161_gb300 as P
    lib = P._lib
    with pytest.raises(P.AF1Error) as e:
        P.rank_for_budget(-1, 4)
    assert e.value.code == -1
    # NULL desc / NULL out / over-budget rank are rejected before any CUDA call
    h = ctypes.c_void_p()
    assert lib.af1_pack_layer(None, None, None, None, None, None, None, None, None, ctypes.byref(h)) == -1
    d = P._Desc(64, 64, 10_000, 0, 0)
    assert lib.af1_pack_layer(ctypes.byref(d), None, None, None, None, None, None, None, None,
                              ctypes.byref(h)) == -4
    assert "exceeds the 1.0-BPW rank" in P.last_error()
    d = P._Desc(64, 64, 10, 0, 7)
    assert lib.af1_pack_layer(ctypes.byref(d), None, None, None, None, None, None, None, None,
                              ctypes.byref(h)) == -1
    d = P._Desc(64, 0, 10, 0, 0)
    assert lib.af1_load_packed_layer(ctypes.byref(d), None, None, None, None, None, None, ctypes.byref(h)) == -1
    assert lib.af1_linear_forward(None, None, 0, 1, None, 0, 0, None, 0, None) == -1
    assert lib.af1_workspace_bytes(None, 1) == -1
    assert lib.af1_workspace_bytes_swiglu(None, 1) == -1
    assert lib.af1_linear_forward_swiglu(None, None, None, 0, 1, None, 0, 0, None, 0, None) == -1
    assert "u is NULL" in P.last_error()
    prm = P._NabfParams(3, 10, 1.0, 0.01, 1e-8, 0, 1, 0)
    assert lib.af1_nabf_factorize(None, 8, 8, 4, None, None, None, None, None, None, None, None, None, None) == -1
    assert lib.af1_nabf_factorize(None, 8, 8, 9, None, None, ctypes.byref(prm), None, None, None, None, None, None,
                                  None) == -1  # r > min(m, n)
    bad = P._NabfParams(3, 10, 0.0, 0.01, 1e-8, 0, 1, 0)  # rho = 0
    assert lib.af1_nabf_factorize(None, 8, 8, 4, None, None, ctypes.byref(bad), None, None, None, None, None, None,
                                  None) == -1
    lib.af1_free(None)  # NULL-safe
    assert P.version().startswith("af1-gb300")


def test_stream_layout_setting():
    _ensure_built()
    import paper_2609_06161_gb300 as P
    assert P.get_stream_layout() == P.AF1_ONE_STREAM  # the default
    try:
        P.set_stream_layout(P.AF1_MANY_STREAMS)
        assert P.get_stream_layout() == P.AF1_MANY_STREAMS
        with pytest.raises(P.AF1Error) as e:
            P.set_stream_layout(2)
        assert e.value.code == -1
        assert P.get_stream_layout() == P.AF1_MANY_STREAMS  # unchanged by the rejected call
    finally:
        P.set_stream_layout(P.AF1_ONE_STREAM)
    assert P.get_stream_layout() == P.AF1_ONE_STREAM
