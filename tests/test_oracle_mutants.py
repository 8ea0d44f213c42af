"""The pins in test_oracle.py must reject plausible mistakes. Each mutant below
is a copy of the oracle forward with one planted error (a dropped term, a
transposed factor, swapped scales, a wrong bit order); the golden fixtures
and closed forms must catch every one. Runs on CPU only."""
import numpy as np
import pytest

from oracle import af1_oracle as O
from tests.golden_io import load


def fwd_ok(U, V, a, s, b, x):
    return O.forward_factored(U, V, a, s, b, x)


def mut_drop_rank_scale(U, V, a, s, b, x):
    return (x * b) @ V @ U.T * a


def mut_transpose_core(U, V, a, s, b, x):
    # uses U for the input side and V for the output side
    return ((x * b) @ U * s) @ V.T * a


def mut_swap_row_col_scales(U, V, a, s, b, x):
    return ((x * a) @ V * s) @ U.T * b


def mut_sign_flip(U, V, a, s, b, x):
    return -(((x * b) @ V * s) @ U.T * a)


def mut_drop_col_scale(U, V, a, s, b, x):
    return ((x @ V) * s) @ U.T * a


MUTANTS = [mut_drop_rank_scale, mut_transpose_core, mut_swap_row_col_scales, mut_sign_flip,
           mut_drop_col_scale]


def golden_cases():
    g = load("worked_example.txt")
    yield [g[k] for k in ("U", "V", "a", "s", "b")], g["W"]
    h = load("nonsymmetric_example.txt")
    for c in ("case1", "case2"):
        yield [h[f"{c}.{k}"] for k in ("U", "V", "a", "s", "b")], h[f"{c}.W"]


def passes_pins(fwd):
    for args, W in golden_cases():
        for j in range(2):
            x = np.zeros((1, 2))
            x[0, j] = 1.0
            if not np.allclose(fwd(*args, x)[0], W[:, j], rtol=0, atol=1e-12):
                return False
    return True


def test_reference_passes():
    assert passes_pins(fwd_ok)


@pytest.mark.parametrize("mutant", MUTANTS, ids=lambda f: f.__name__)
def test_mutant_is_caught(mutant):
    assert not passes_pins(mutant)


def test_bit_order_mutant_is_caught():
    g = load("packed_words.txt")
    S = np.asarray(g["row3.signs"], dtype=np.int64).reshape(1, -1)

    def pack_msb_first(S):
        w = O.pack_rows(S)
        rev = np.zeros_like(w)
        for i in range(32):
            rev |= ((w >> np.uint32(i)) & np.uint32(1)) << np.uint32(31 - i)
        return rev

    assert not np.array_equal(pack_msb_first(S)[0].astype(np.int64),
                              np.asarray(g["row3.words"], dtype=np.int64))
