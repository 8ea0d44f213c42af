"""HiSA budget arithmetic (host functions of the C ABI) against the oracle,
and the oracle against closed forms. No GPU needed."""
import math

import numpy as np
import pytest

from oracle import af1_oracle as O


@pytest.fixture(scope="module")
def P():
    from tests.test_abi_host import _ensure_built
    _ensure_built()
    import paper_2609_06161_gb300 as P
    return P


# -- oracle pins -------------------------------------------------------------

def test_layer_softmax_closed_forms():
    assert O.hisa_layer_budgets([0.0, math.log(3.0)], 4.0, 1.0) == pytest.approx([1.0, 3.0], rel=1e-15)
    assert O.hisa_layer_budgets([0.7] * 5, 5.0, 0.3) == pytest.approx([1.0] * 5, rel=1e-15)
    b = O.hisa_layer_budgets([0.1, 0.5, -2.0, 3.0], 32.0, 1.0)
    assert sum(b) == pytest.approx(32.0, rel=1e-14)
    # tau -> infinity: uniform; tau -> 0: all budget on the best layer
    assert O.hisa_layer_budgets([0.1, 0.5, -2.0], 3.0, 1e9) == pytest.approx([1.0] * 3, rel=1e-6)
    assert O.hisa_layer_budgets([0.1, 0.5, -2.0], 3.0, 1e-4) == pytest.approx([0.0, 3.0, 0.0], abs=1e-12)


def test_mad_z_hand_values():
    # median 3, absolute deviations 2, 1, 0, 1, 97 -> MAD 1
    z = O.mad_z([1.0, 2.0, 3.0, 4.0, 100.0], 0.0)
    assert z == pytest.approx([-2 / 1.4826, -1 / 1.4826, 0.0, 1 / 1.4826, 97 / 1.4826], rel=1e-15)
    # even count: median of the middle pair
    z = O.mad_z([1.0, 3.0, 5.0, 11.0], 0.0)  # median 4, deviations 3 1 1 7 -> MAD 2
    assert z == pytest.approx([-3 / 2.9652, -1 / 2.9652, 1 / 2.9652, 7 / 2.9652], rel=1e-15)


def test_module_budgets_closed_forms():
    params = [4096 * 4096, 1024 * 4096, 1024 * 4096, 4096 * 4096, 14336 * 4096, 14336 * 4096, 4096 * 14336]
    g = np.random.default_rng(0)
    pd, pm = g.random(7).tolist(), g.random(7).tolist()
    b = O.hisa_module_budgets(pd, pm, params, 1.0, 0.2, 1e-8)
    # the parameter-weighted mean is the layer budget
    assert sum(p * x for p, x in zip(params, b)) / sum(params) == pytest.approx(1.0, rel=1e-14)
    # alpha = 0: every density 1, every module gets the layer budget
    assert O.hisa_module_budgets(pd, pm, params, 1.25, 0.0, 1e-8) == pytest.approx([1.25] * 7, rel=1e-15)
    # scores at the median of both distortions: z = 0, P = 1/2, v = 3/4
    b = O.hisa_module_budgets([1.0, 2.0, 3.0], [5.0, 6.0, 7.0], [10, 10, 10], 2.0, 1.0, 0.0)
    v_mid = 1 - 0.25
    assert b[1] == pytest.approx(2.0 * 30 * (v_mid / 10) / sum(10 * w for w in [
        (1 - (1 - 1 / (1 + math.exp(1 / 1.4826))) ** 2) / 10, v_mid / 10,
        (1 - (1 - 1 / (1 + math.exp(-1 / 1.4826))) ** 2) / 10]), rel=1e-14)


def test_budget_to_rank_paper_value():
    # App. "Budget-to-rank conversion" at 1.0 BPW, dominant bits: 4096^2 -> 2048
    assert O.budget_to_rank(1.0, 4096, 4096) == 2048
    assert O.budget_to_rank(1.0, 4096, 4096) == O.rank_dominant_bits(4096, 4096, 1)
    assert O.budget_to_rank(0.0, 10, 10) == 1 and O.budget_to_rank(1e9, 10, 10) == 32768


# -- the library against the oracle ------------------------------------------

def test_library_matches_oracle(P):
    g = np.random.default_rng(1)
    for L in (1, 2, 7, 32):
        phi = (g.normal(0, 0.3, L)).tolist()
        for tau in (0.5, 1.0, 3.0):
            lib = P.hisa_layer_budgets(phi, float(L), tau)
            assert lib == pytest.approx(O.hisa_layer_budgets(phi, float(L), tau), rel=1e-13)
    for N in (1, 2, 3, 7):
        pd, pm = g.random(N).tolist(), (g.random(N) * 10).tolist()
        params = g.integers(1, 1 << 26, N).tolist()
        for alpha in (0.0, 0.2, 1.0):
            lib = P.hisa_module_budgets(pd, pm, params, 1.0, alpha, 1e-8)
            assert lib == pytest.approx(O.hisa_module_budgets(pd, pm, params, 1.0, alpha, 1e-8), rel=1e-12)
    for (b, m, n) in [(1.0, 4096, 4096), (0.8, 1024, 4096), (1.3, 14336, 4096), (2.5, 8192, 28672), (0.0, 7, 9)]:
        assert P.budget_to_rank(b, m, n) == O.budget_to_rank(b, m, n)


def test_library_rejects_bad_arguments(P):
    with pytest.raises(P.AF1Error):
        P.hisa_layer_budgets([0.1, 0.2], 2.0, 0.0)
    with pytest.raises(P.AF1Error):
        P.hisa_layer_budgets([0.1, float("nan")], 2.0, 1.0)
    with pytest.raises(P.AF1Error):
        P.hisa_module_budgets([0.1], [0.2], [0], 1.0)
    with pytest.raises(P.AF1Error):
        P.budget_to_rank(-1.0, 4, 4)
