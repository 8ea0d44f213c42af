"""Pins for the CPU oracle: paper-printed values, closed forms, brute force and
exact integer search. None of these call the CUDA path."""
import itertools
from fractions import Fraction

import numpy as np
import pytest

import synth
from oracle import af1_oracle as O
from tests.golden_io import load

CONFIG_SHAPES = {
    # (d_out, d_in): r from the exact 1.0-BPW storage rule
    (4096, 4096): 2028,
    (1024, 4096): 800,
    (14336, 4096): 3167,
    (4096, 14336): 3167,
    (8192, 8192): 4076,
    (1024, 8192): 892,
    (28672, 8192): 6352,
    (8192, 28672): 6352,
}


# --------------------------------------------------------------------------
# Worked example printed in the paper (App., Eq. double_example)
# --------------------------------------------------------------------------

def test_worked_example_matches_paper():
    g = load("worked_example.txt")
    W = O.reconstruct_dense(g["U"], g["V"], g["a"], g["s"], g["b"])
    np.testing.assert_array_equal(W, g["W"])
    assert np.linalg.det(W) == pytest.approx(float(g["det"][0] if np.ndim(g["det"]) else g["det"]))


def test_worked_example_forward_unit_vectors():
    g = load("worked_example.txt")
    for j in range(2):
        x = np.zeros((1, 2))
        x[0, j] = 1.0
        y_f = O.forward_factored(g["U"], g["V"], g["a"], g["s"], g["b"], x)
        np.testing.assert_array_equal(y_f[0], g["W"][:, j])


@pytest.mark.parametrize("case", ["case1", "case2"])
def test_nonsymmetric_examples(case):
    g = load("nonsymmetric_example.txt")
    args = [g[f"{case}.{k}"] for k in ("U", "V", "a", "s", "b")]
    W = O.reconstruct_dense(*args)
    np.testing.assert_array_equal(W, g[f"{case}.W"])
    for j in range(2):
        x = np.zeros((1, 2))
        x[0, j] = 1.0
        np.testing.assert_array_equal(O.forward_factored(*args, x)[0], g[f"{case}.W"][:, j])
        np.testing.assert_array_equal(O.forward_dense(W, x)[0], g[f"{case}.W"][:, j])


# --------------------------------------------------------------------------
# Brute force: every sign pattern of a 2 x 2 x 2 layer against the path sum
# --------------------------------------------------------------------------

def test_bruteforce_all_sign_patterns_2x2x2():
    rng = np.random.default_rng(7)
    a = rng.uniform(0.5, 2.0, 2)
    b = rng.uniform(0.5, 2.0, 2)
    s = rng.uniform(-1.0, 1.0, 2)
    x = rng.normal(size=(3, 2))
    for bits in itertools.product((-1, 1), repeat=8):
        U = np.array(bits[:4]).reshape(2, 2)
        V = np.array(bits[4:]).reshape(2, 2)
        W = O.reconstruct_dense(U, V, a, s, b)
        for i in range(2):
            for j in range(2):
                # triple loop written straight from the path-sum form
                ref = 0.0
                for k in range(2):
                    ref += s[k] * U[i, k] * V[j, k]
                ref *= a[i] * b[j]
                assert W[i, j] == pytest.approx(ref, abs=1e-15)
                assert O.reconstruct_entry(U, V, a, s, b, i, j) == pytest.approx(ref, abs=1e-15)
        y = O.forward_factored(U, V, a, s, b, x)
        y_naive = np.array([[sum(W[i, j] * x[t, j] for j in range(2)) for i in range(2)]
                            for t in range(3)])
        np.testing.assert_allclose(y, y_naive, rtol=0, atol=1e-14)


def test_bruteforce_random_small_shapes_triple_loop():
    rng = np.random.default_rng(11)
    for (m, n, r) in [(3, 5, 2), (5, 3, 4), (7, 6, 1), (4, 9, 3)]:
        U = np.where(rng.integers(0, 2, (m, r)) == 1, 1, -1)
        V = np.where(rng.integers(0, 2, (n, r)) == 1, 1, -1)
        a, s, b = rng.normal(size=m), rng.normal(size=r), rng.normal(size=n)
        W = O.reconstruct_dense(U, V, a, s, b)
        for i in range(m):
            for j in range(n):
                acc = 0.0
                for k in range(r):
                    acc += s[k] * U[i][k] * V[j][k]
                assert W[i, j] == pytest.approx(a[i] * b[j] * acc, rel=1e-13, abs=1e-13)


# --------------------------------------------------------------------------
# Closed forms
# --------------------------------------------------------------------------

def sylvester(k):
    H = np.array([[1]])
    for _ in range(k):
        H = np.block([[H, H], [H, -H]])
    return H


@pytest.mark.parametrize("k", [1, 3, 5, 7])
def test_hadamard_identity(k):
    """U = V = H (Sylvester), s = 1/N: U Diag(s) V^T = H H^T / N = I, so the
    layer reduces to y_i = a_i b_i x_i exactly."""
    N = 2 ** k
    H = sylvester(k)
    rng = np.random.default_rng(k)
    a, b = rng.normal(size=N), rng.normal(size=N)
    s = np.full(N, 1.0 / N)
    W = O.reconstruct_dense(H, H, a, s, b)
    np.testing.assert_allclose(W, np.diag(a * b), rtol=0, atol=1e-14)
    x = rng.normal(size=(2, N))
    np.testing.assert_allclose(O.forward_factored(H, H, a, s, b, x), x * (a * b)[None, :],
                               rtol=1e-13, atol=1e-14)


def test_rank_one_is_outer_product():
    rng = np.random.default_rng(3)
    m, n = 6, 9
    U = np.where(rng.integers(0, 2, (m, 1)) == 1, 1, -1)
    V = np.where(rng.integers(0, 2, (n, 1)) == 1, 1, -1)
    a, b = rng.normal(size=m), rng.normal(size=n)
    s = np.array([0.37])
    W = O.reconstruct_dense(U, V, a, s, b)
    np.testing.assert_allclose(W, 0.37 * np.outer(a * U[:, 0], b * V[:, 0]), rtol=1e-14, atol=0)


def test_dense_equals_factored_random():
    rng = np.random.default_rng(5)
    for (m, n, r, T) in [(64, 48, 40, 3), (130, 257, 97, 5), (256, 256, 120, 1)]:
        U = np.where(rng.integers(0, 2, (m, r)) == 1, 1, -1)
        V = np.where(rng.integers(0, 2, (n, r)) == 1, 1, -1)
        a, s, b = rng.normal(size=m), rng.normal(size=r), rng.normal(size=n)
        x = rng.normal(size=(T, n))
        yd = O.forward_dense(O.reconstruct_dense(U, V, a, s, b), x)
        yf = O.forward_factored(U, V, a, s, b, x)
        assert O.rowwise_rel_err(yf, yd) < 1e-12
        rows = rng.choice(m, 7, replace=False)
        np.testing.assert_allclose(O.forward_factored(U, V, a, s, b, x, rows=rows), yf[:, rows],
                                   rtol=1e-14, atol=1e-14)


def test_linearity_in_x_and_scales():
    rng = np.random.default_rng(9)
    m, n, r = 20, 30, 12
    U = np.where(rng.integers(0, 2, (m, r)) == 1, 1, -1)
    V = np.where(rng.integers(0, 2, (n, r)) == 1, 1, -1)
    a, s, b = rng.normal(size=m), rng.normal(size=r), rng.normal(size=n)
    x1, x2 = rng.normal(size=(2, n)), rng.normal(size=(2, n))
    f = lambda a_, s_, b_, x_: O.forward_factored(U, V, a_, s_, b_, x_)
    np.testing.assert_allclose(f(a, s, b, 2 * x1 - 3 * x2), 2 * f(a, s, b, x1) - 3 * f(a, s, b, x2),
                               rtol=1e-12, atol=1e-12)
    s2 = rng.normal(size=r)
    np.testing.assert_allclose(f(a, s + s2, b, x1), f(a, s, b, x1) + f(a, s2, b, x1), rtol=1e-12, atol=1e-12)
    a2 = rng.normal(size=m)
    np.testing.assert_allclose(f(a + a2, s, b, x1), f(a, s, b, x1) + f(a2, s, b, x1), rtol=1e-12, atol=1e-12)
    b2 = rng.normal(size=n)
    np.testing.assert_allclose(f(a, s, b + b2, x1), f(a, s, b, x1) + f(a, s, b2, x1), rtol=1e-12, atol=1e-12)


def test_integer_inputs_give_exact_integers():
    """Unit scales and integer activations: the exact result is an integer
    matrix product, reproduced exactly by brute force."""
    rng = np.random.default_rng(13)
    m, n, r = 40, 50, 30
    U = np.where(rng.integers(0, 2, (m, r)) == 1, 1, -1)
    V = np.where(rng.integers(0, 2, (n, r)) == 1, 1, -1)
    x = rng.integers(-2, 3, (3, n))
    y = O.forward_factored(U, V, np.ones(m), np.ones(r), np.ones(n), x)
    ref = x.astype(np.int64) @ V.astype(np.int64) @ U.T.astype(np.int64)
    np.testing.assert_array_equal(y, ref.astype(np.float64))


# --------------------------------------------------------------------------
# Packing
# --------------------------------------------------------------------------

@pytest.mark.parametrize("row", ["row1", "row2", "row3"])
def test_pack_hand_computed_words(row):
    g = load("packed_words.txt")
    S = np.asarray(g[f"{row}.signs"], dtype=np.int64).reshape(1, -1)
    words = O.pack_rows(S)
    np.testing.assert_array_equal(words[0].astype(np.int64), np.asarray(g[f"{row}.words"], dtype=np.int64))
    np.testing.assert_array_equal(O.unpack_rows(words, S.shape[1]), S)


@pytest.mark.parametrize("R,C", [(1, 1), (3, 31), (5, 32), (7, 33), (4, 127), (2, 128), (9, 129), (16, 2028)])
def test_pack_roundtrip_and_padding(R, C):
    rng = np.random.default_rng(R * 1000 + C)
    S = np.where(rng.integers(0, 2, (R, C)) == 1, 1, -1).astype(np.int8)
    w = O.pack_rows(S)
    assert w.dtype == np.uint32
    assert w.shape == (R, 4 * ((C + 127) // 128))
    assert O.padding_is_zero(w, C)
    np.testing.assert_array_equal(O.unpack_rows(w, C), S)
    # word-level identity in the other direction: unpack -> pack
    np.testing.assert_array_equal(O.pack_rows(O.unpack_rows(w, C)), w)


def test_pack_V_is_transposed_B():
    rng = np.random.default_rng(2)
    n, r = 70, 9
    V = np.where(rng.integers(0, 2, (n, r)) == 1, 1, -1).astype(np.int8)
    Vw = O.pack_V(V)
    assert Vw.shape == (r, 4)
    for k in range(r):
        for j in range(n):
            bit = (int(Vw[k, j // 32]) >> (j % 32)) & 1
            assert bit == (1 if V[j, k] == 1 else 0)
    np.testing.assert_array_equal(O.unpack_V(Vw, n), V)


def test_pack_rejects_non_signs():
    with pytest.raises(ValueError):
        O.pack_rows(np.array([[1, 0, -1]]))
    with pytest.raises(ValueError):
        O.pack_rows(np.array([[1, 2]]))


def test_forward_from_packed_matches_signs():
    from synth import layer_signs
    d = layer_signs(21, 96, 160, 70, 3)
    Uw, Vw = O.pack_U(d["U"]), O.pack_V(d["V"])
    y = O.forward_from_packed(Uw, Vw, d["a"], d["s"], d["b"], d["x"], 96, 160, 70)
    yd = O.forward_dense(
        O.reconstruct_dense(d["U"], d["V"], O.f16_bits_to_f64(d["a"]), O.f16_bits_to_f64(d["s"]),
                            O.f16_bits_to_f64(d["b"])),
        O.f16_bits_to_f64(d["x"]).reshape(3, 160))
    assert O.rowwise_rel_err(y, yd) < 1e-12


# --------------------------------------------------------------------------
# FP16 widening
# --------------------------------------------------------------------------

def test_f16_widening_exact():
    bits = np.array([0x3C00, 0xC000, 0x0001, 0x7BFF, 0x3555, 0x8000], dtype=np.uint16)
    v = O.f16_bits_to_f64(bits)
    assert v[0] == 1.0 and v[1] == -2.0 and v[2] == 2.0 ** -24 and v[3] == 65504.0
    assert v[4] == 1365 / 4096  # 0x3555: exponent 13 -> 2^-2 * (1 + 341/1024)
    assert v[5] == 0.0 and np.signbit(v[5])


def test_bf16_widening_exact():
    # BF16 = the upper half of an FP32: 1 sign, 8 exponent (bias 127), 7 mantissa bits.
    bits = np.array([0x3F80, 0xC000, 0x3C23, 0x7F7F, 0x0001, 0x8000], dtype=np.uint16)
    v = O.bf16_bits_to_f64(bits)
    assert v[0] == 1.0 and v[1] == -2.0
    assert v[2] == 163 / 16384  # exponent 120 -> 2^-7 * (1 + 35/128)
    assert v[3] == 255 * 2.0 ** 120  # largest finite: 2^127 * (1 + 127/128)
    assert v[4] == 2.0 ** -133  # smallest subnormal: 2^-126 * 2^-7
    assert v[5] == 0.0 and np.signbit(v[5])


def test_forward_bf16_scales_equal_f16_scales_of_equal_value():
    """Scales whose BF16 and FP16 patterns hold the same values (dyadic
    numbers with few significant bits) give the same forward; each of a, s, b
    is decoded as BF16 (a pattern read as FP16 instead would change it)."""
    g = synth.rng(5)
    m, n, r, T = 9, 14, 6, 2
    U, V = synth.signs(g, m, r), synth.signs(g, n, r)
    vals = [0.5, 0.25, 1.5, 0.125, 2.0, 0.75]
    def pick(k):
        v = np.array([vals[i % len(vals)] for i in range(k)], dtype=np.float32)
        f16 = v.astype(np.float16).view(np.uint16)
        b16 = (v.view(np.uint32) >> np.uint32(16)).astype(np.uint16)
        return f16, b16
    (a16, ab), (s16, sb), (b16_, bb) = pick(m), pick(r), pick(n)
    X = synth.activations_f16(g, T, n)
    Uw, Vw = O.pack_U(U), O.pack_V(V)
    y16 = O.forward_from_packed(Uw, Vw, a16, s16, b16_, X, m, n, r)
    ybf = O.forward_from_packed(Uw, Vw, ab, sb, bb, X, m, n, r, scale_dtype="bf16")
    np.testing.assert_array_equal(y16, ybf)
    assert not np.array_equal(O.bf16_bits_to_f64(ab), O.f16_bits_to_f64(ab))


# --------------------------------------------------------------------------
# Storage accounting and the rank rule (App. "Effective Bit-Width")
# --------------------------------------------------------------------------

@pytest.mark.parametrize("shape,r_expected", sorted(CONFIG_SHAPES.items()))
def test_rank_rule_exhaustive(shape, r_expected):
    m, n = shape
    r = O.rank_for_budget(m, n, 1)
    assert r == r_expected
    # exhaustive search over every rank up to the dense count, from the
    # storage formula alone
    budget = m * n
    best = max(k for k in range(0, min(m, n) + 1) if O.storage_bits(m, n, k) <= budget)
    assert r == best
    assert O.storage_bits(m, n, r) <= budget < O.storage_bits(m, n, r + 1)
    assert O.bpw([(m, n, r)]) <= 1 < O.bpw([(m, n, r + 1)])


def test_storage_formula_hand_value():
    # 4096 x 4096 at r = 2028: 2028 * 8192 + 16 * (4096 + 2028 + 4096)
    assert O.storage_bits(4096, 4096, 2028) == 2028 * 8192 + 16 * 10220 == 16777216 - 320
    assert O.bpw([(4096, 4096, 2028)]) == Fraction(16777216 - 320, 16777216)


def test_rank_rule_other_budgets():
    for bpw in (Fraction(5, 2), Fraction(1, 2), 2):
        for (m, n) in [(4096, 4096), (1024, 4096), (300, 700)]:
            r = O.rank_for_budget(m, n, bpw)
            B = Fraction(bpw) * m * n
            assert O.storage_bits(m, n, r) <= B < O.storage_bits(m, n, r + 1)
    assert O.rank_for_budget(4, 4, 1) == 0  # 16 weights cannot carry the scales


def test_paper_dominant_bit_rule():
    # App. A.3 rounds b * d_out * d_in / (d_out + d_in); at 4096^2 and 1 BPW
    # that is exactly 2048, which overshoots the full-storage budget.
    assert O.rank_dominant_bits(4096, 4096, 1) == 2048
    assert O.storage_bits(4096, 4096, 2048) > 4096 * 4096
    assert O.rank_dominant_bits(1024, 4096, 1) == round(1024 * 4096 / 5120)


# --------------------------------------------------------------------------
# Error metric
# --------------------------------------------------------------------------

def test_rowwise_rel_err():
    ref = np.array([[1.0, -4.0, 2.0], [0.0, 0.0, 0.0]])
    y = ref + np.array([[0.0, 0.004, 0.0], [0.0, 1e-3, 0.0]])
    assert O.rowwise_rel_err(y, ref) == pytest.approx(1e-3)
    assert O.rowwise_rel_err(ref, ref) == 0.0
    assert O.rowwise_rel_err(np.zeros((0, 3)), np.zeros((0, 3))) == 0.0


# ---- SwiGLU input of a down projection (oracle side) -----------------------

def test_silu_against_the_tanh_form_and_the_odd_part():
    # SiLU(z) = z sigmoid(z) = (z / 2) (1 + tanh(z / 2)), and SiLU(z) - SiLU(-z) = z
    # because sigmoid(z) + sigmoid(-z) = 1.
    z = np.linspace(-30.0, 30.0, 2001)
    # (the tanh form cancels for z << 0: compare absolutely there)
    np.testing.assert_allclose(O.silu_f64(z), 0.5 * z * (1.0 + np.tanh(0.5 * z)), rtol=1e-13, atol=1e-14)
    np.testing.assert_allclose(O.silu_f64(z) - O.silu_f64(-z), z, rtol=1e-13, atol=1e-13)
    assert O.silu_f64(0.0) == 0.0
    assert O.silu_f64(1.0) == pytest.approx(0.7310585786300049, rel=1e-15)   # 1 / (1 + 1/e)
    assert O.silu_f64(-1e4) == 0.0 or abs(O.silu_f64(-1e4)) < 1e-300          # no overflow to NaN


def test_swiglu_f16_rounds_once():
    g = np.array([0.0, 1.0, -1.0, 2.0, 20.0, -20.0, 3.0, 65504.0], dtype=np.float16)
    u = np.array([5.0, 1.0, 1.0, -0.5, 2.0, 1.0, 0.0, 1.0], dtype=np.float16)
    h = O.swiglu_f16(g.view(np.uint16), u.view(np.uint16)).view(np.float16).astype(np.float64)
    ref = [0.0,
           float(np.float16(0.7310585786300049)),        # SiLU(1)
           float(np.float16(-0.2689414213699951)),       # SiLU(-1) = SiLU(1) - 1
           float(np.float16(-0.5 * 1.7615941559557649)),  # SiLU(2) * -0.5
           40.0,                                           # SiLU(20) = 20 - 4e-8 -> 20, times 2
           float(np.float16(-20.0 / (1.0 + np.exp(20.0)))),  # about -4.1e-8: a subnormal
           0.0,
           65504.0]                                        # SiLU(65504) = 65504 exactly in FP16
    np.testing.assert_array_equal(h, ref)
    # Sign symmetry of round to nearest: negating u negates h.
    hn = O.swiglu_f16(g.view(np.uint16), (-u).view(np.uint16)).view(np.float16).astype(np.float64)
    np.testing.assert_array_equal(hn, -h)
