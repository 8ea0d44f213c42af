"""Plain CPU oracle for the AF1 binary-factorized linear layer (FP64).

TEST INFRASTRUCTURE ONLY. Nothing on the product path may import, call or
execute this module: only ``tests/``, ``__graft_entry__.smoke()`` and the
CPU-baseline / reference legs of ``bench.py`` use it. It shares no code with
the CUDA path (no headers, helpers, tables or constant generators) and does
not import the package.

What it computes (AF1, Sec. 3.1, Eq. final_reconstruction; App. "Double-factor
binary representation", Eq. double_factor_equiv and Eq. binary_paths):

    W_hat = Diag(a) . A_pm1 . Diag(m) . B_pm1 . Diag(b)        (m = m1 * m2)
    W_hat[i, j] = a_i * b_j * sum_k m_k * A[i, k] * B[k, j]
    y = x . W_hat^T   (a linear layer, W_hat is d_out x d_in)

Notation used here: U = A_pm1 (d_out x r), V = B_pm1^T (d_in x r), s = the
merged rank scale m (renamed so that it does not clash with the dimension
m = d_out), n = d_in. All scale vectors and activations arrive as FP16 bit
patterns and are widened to float64 exactly; every product and sum below is
FP64.

Storage accounting follows App. "Effective Bit-Width", Eq. app_af1_memory and
Eq. app_af1_bpw; the rank rule is the exact inversion of that storage count
(the paper's App. A.3 rounds the dominant bits only; both are provided).

Packing layout (the paper gives none; reading fixed here): each factor is
packed along its contraction axis, LSB first, bit = 1 <=> +1, bit = 0 <=> -1,
32 signs per uint32 word, each row padded to a multiple of 4 words (16 bytes)
with zero bits.
  * U (d_out x r): row i holds U[i, 0..r-1]          -> d_out x W(r) words
  * V (d_in x r):  row k holds V[0..d_in-1, k] = B[k, :] -> r x W(d_in) words
where W(c) = 4 * ceil(c / 128).

Parity pins: every function here is checked in tests/test_oracle.py against
values the paper prints (the 2x2 worked example of App. "Strictly richer
magnitude patterns"), closed forms (Sylvester-Hadamard identity, rank-1 outer
product), brute force over every sign pattern of a 2x2x2 layer, exact integer
search for the storage rule, and hand-computed packed words.
"""
from __future__ import annotations

from fractions import Fraction
import math

import numpy as np

WORD_BITS = 32
ROW_ALIGN_WORDS = 4  # rows padded to 16 bytes


# ---------------------------------------------------------------------------
# Storage accounting (App. "Effective Bit-Width", Eq. app_af1_memory/bpw)
# ---------------------------------------------------------------------------

def storage_bits(d_out: int, d_in: int, r: int) -> int:
    """Deployable bits of one AF1 matrix: r(d_out + d_in) sign bits plus three
    16-bit scale vectors of lengths d_out, r, d_in (Eq. app_af1_memory)."""
    return r * (d_out + d_in) + 16 * (d_out + r + d_in)


def bpw(layers) -> Fraction:
    """Effective bits per weight over a set of (d_out, d_in, r) matrices
    (Eq. app_af1_bpw), as an exact fraction."""
    num = sum(storage_bits(o, i, r) for (o, i, r) in layers)
    den = sum(o * i for (o, i, _r) in layers)
    return Fraction(num, den)


def rank_for_budget(d_out: int, d_in: int, budget_bpw=1) -> int:
    """Largest r whose exact storage (Eq. app_af1_memory) fits the budget
    budget_bpw * d_out * d_in. Reading of the paper: the budget is a hard cap
    on the full storage, scales included, so M(r) <= budget < M(r + 1).
    Solving r(d_out + d_in) + 16(d_out + r + d_in) <= B for integer r gives
    r = floor((B - 16(d_out + d_in)) / (d_out + d_in + 16)). Returns 0 when
    not even rank 1 fits."""
    B = Fraction(budget_bpw) * d_out * d_in
    r = (B - 16 * (d_out + d_in)) / (d_out + d_in + 16)
    return max(0, math.floor(r))


def rank_dominant_bits(d_out: int, d_in: int, budget_bpw=1) -> int:
    """The paper's printed conversion (App. A.3, "Budget-to-rank conversion"):
    Round(b * d_out * d_in / (d_out + d_in)), counting sign bits only.
    Round-half-up is used for ties (the paper does not say)."""
    v = Fraction(budget_bpw) * d_out * d_in / (d_out + d_in)
    return math.floor(v + Fraction(1, 2))


# ---------------------------------------------------------------------------
# Packing (layout fixed above)
# ---------------------------------------------------------------------------

def words_per_row(cols: int) -> int:
    """uint32 words per packed row of `cols` signs, padded to 16 bytes."""
    return ROW_ALIGN_WORDS * ((cols + 127) // 128)


def pack_rows(S: np.ndarray) -> np.ndarray:
    """Pack an R x C matrix of +-1 into R x words_per_row(C) uint32 words:
    bit (c mod 32) of word (c div 32) of row i is 1 iff S[i, c] == +1."""
    S = np.asarray(S)
    if S.ndim != 2:
        raise ValueError("expected a 2-D sign matrix")
    if not np.all((S == 1) | (S == -1)):
        raise ValueError("sign matrix entries must be exactly +1 or -1")
    R, C = S.shape
    W = words_per_row(C)
    bits = np.zeros((R, W * WORD_BITS), dtype=np.uint64)
    bits[:, :C] = (S == 1)
    weights = np.uint64(1) << np.arange(WORD_BITS, dtype=np.uint64)
    words = (bits.reshape(R, W, WORD_BITS) * weights).sum(axis=2)
    return words.astype(np.uint32)


def unpack_rows(words: np.ndarray, cols: int) -> np.ndarray:
    """Inverse of pack_rows: R x W words -> R x cols int8 matrix of +-1."""
    words = np.asarray(words, dtype=np.uint32)
    R, W = words.shape
    if W * WORD_BITS < cols:
        raise ValueError("not enough words for the requested columns")
    shifts = np.arange(WORD_BITS, dtype=np.uint32)
    bits = (words[:, :, None] >> shifts) & np.uint32(1)
    bits = bits.reshape(R, W * WORD_BITS)[:, :cols]
    return np.where(bits == 1, 1, -1).astype(np.int8)


def pack_U(U: np.ndarray) -> np.ndarray:
    """U = A_pm1 (d_out x r) packed along r: d_out x words_per_row(r)."""
    return pack_rows(U)


def pack_V(V: np.ndarray) -> np.ndarray:
    """V = B_pm1^T (d_in x r) packed along d_in: row k is B[k, :], so the
    result is r x words_per_row(d_in)."""
    return pack_rows(np.asarray(V).T)


def unpack_U(Uw: np.ndarray, r: int) -> np.ndarray:
    return unpack_rows(Uw, r)


def unpack_V(Vw: np.ndarray, d_in: int) -> np.ndarray:
    """Returns V (d_in x r) from its r x W packed rows."""
    return unpack_rows(Vw, d_in).T


def padding_is_zero(words: np.ndarray, cols: int) -> bool:
    """True iff every bit at column >= cols of every packed row is zero."""
    words = np.asarray(words, dtype=np.uint32)
    R, W = words.shape
    shifts = np.arange(WORD_BITS, dtype=np.uint32)
    bits = ((words[:, :, None] >> shifts) & np.uint32(1)).reshape(R, W * WORD_BITS)
    return not bits[:, cols:].any()


# ---------------------------------------------------------------------------
# FP16 inputs
# ---------------------------------------------------------------------------

def f16_bits_to_f64(h) -> np.ndarray:
    """FP16 bit patterns (uint16) -> float64, exact."""
    h = np.ascontiguousarray(np.asarray(h, dtype=np.uint16))
    return h.view(np.float16).astype(np.float64)


def bf16_bits_to_f64(h) -> np.ndarray:
    """BF16 bit patterns (uint16) -> float64, exact: a BF16 value is the
    FP32 value whose upper 16 bits are the pattern and lower 16 bits zero
    (1 sign, 8 exponent, 7 mantissa bits; the paper's scale type)."""
    h = np.ascontiguousarray(np.asarray(h, dtype=np.uint16))
    return (h.astype(np.uint32) << np.uint32(16)).view(np.float32).astype(np.float64)


def f64_to_f16_bits(v) -> np.ndarray:
    """float64 -> FP16 bit patterns, rounded once to nearest (ties to even);
    beyond the FP16 range the result is +-inf."""
    with np.errstate(over="ignore"):
        return np.asarray(v, dtype=np.float64).astype(np.float16).view(np.uint16)


# ---------------------------------------------------------------------------
# SwiGLU input of a down projection (the MLP of the LLaMA models the paper
# compresses: h = SiLU(x W_gate^T) * (x W_up^T), SiLU(z) = z * sigmoid(z)).
# Not part of AF1 itself; the fused entry point takes h from the gate and up
# outputs.
# ---------------------------------------------------------------------------

def silu_f64(z) -> np.ndarray:
    """SiLU(z) = z / (1 + e^-z) in float64."""
    z = np.asarray(z, dtype=np.float64)
    with np.errstate(over="ignore"):
        return z / (1.0 + np.exp(-z))


def swiglu_f16(g_h, u_h) -> np.ndarray:
    """h = SiLU(g) * u from FP16 bit patterns g and u (same shape), in
    float64, rounded once to FP16: the activations the down projection sees.
    Returns FP16 bit patterns."""
    g = f16_bits_to_f64(g_h)
    u = f16_bits_to_f64(u_h)
    return f64_to_f16_bits(silu_f64(g) * u).reshape(np.shape(g_h))


# ---------------------------------------------------------------------------
# Reconstruction and forward (Eq. double_factor_equiv, Eq. binary_paths)
# ---------------------------------------------------------------------------

def reconstruct_dense(U, V, a, s, b) -> np.ndarray:
    """W_hat = Diag(a) U Diag(s) V^T Diag(b), all FP64 (Eq. double_factor_equiv
    with A_pm1 = U and B_pm1 = V^T). U: d_out x r, V: d_in x r, a: d_out,
    s: r, b: d_in (float64 or ints). Returns d_out x d_in."""
    U = np.asarray(U, dtype=np.float64)
    V = np.asarray(V, dtype=np.float64)
    a = np.asarray(a, dtype=np.float64)
    s = np.asarray(s, dtype=np.float64)
    b = np.asarray(b, dtype=np.float64)
    core = (U * s[None, :]) @ V.T          # U Diag(s) B, B = V^T
    return a[:, None] * core * b[None, :]


def reconstruct_entry(U, V, a, s, b, i: int, j: int) -> float:
    """One entry by the path-sum form (Eq. binary_paths):
    a_i b_j sum_k s_k U[i,k] V[j,k]. Plain Python loop, for tiny cases."""
    acc = 0.0
    for k in range(len(s)):
        acc += float(s[k]) * float(U[i][k]) * float(V[j][k])
    return float(a[i]) * float(b[j]) * acc


def forward_dense(W_hat, X) -> np.ndarray:
    """y = X W_hat^T for X of shape (T, d_in) (a linear layer)."""
    return np.asarray(X, dtype=np.float64) @ np.asarray(W_hat, dtype=np.float64).T


def forward_factored(U, V, a, s, b, X, rows=None) -> np.ndarray:
    """The same product evaluated right to left without forming W_hat:
    z = b * x;  t = V^T z  (t_k = sum_j B[k, j] z_j);  u = U (s * t);
    y = a * u. X: (T, d_in). If `rows` is given, only those output columns
    of y (rows of W_hat) are computed; t is always computed in full."""
    X = np.asarray(X, dtype=np.float64)
    b = np.asarray(b, dtype=np.float64)
    s = np.asarray(s, dtype=np.float64)
    a = np.asarray(a, dtype=np.float64)
    z = X * b[None, :]
    t = z @ np.asarray(V, dtype=np.float64)            # (T, r)
    st = t * s[None, :]
    if rows is None:
        Uf = np.asarray(U, dtype=np.float64)
        return (st @ Uf.T) * a[None, :]
    rows = np.asarray(rows)
    Uf = np.asarray(U, dtype=np.float64)[rows]
    return (st @ Uf.T) * a[rows][None, :]


def forward_from_packed(Uw, Vw, a_h, s_h, b_h, X_h, d_out, d_in, r, rows=None, scale_dtype="f16"):
    """Full oracle forward from the deployable format: canonical packed words
    plus FP16 bit patterns of a (d_out), s (r), b (d_in) and X (T x d_in)
    (scale_dtype="bf16": a, s, b are BF16 bit patterns instead). Unpacks the
    signs, widens everything to FP64 exactly and evaluates forward_factored.
    Returns float64 (T x d_out), or (T x len(rows))."""
    U = unpack_U(Uw, r)
    if U.shape[0] != d_out:
        raise ValueError("U rows != d_out")
    V = unpack_V(Vw, d_in)
    if V.shape[1] != r:
        raise ValueError("V rank mismatch")
    dec = {"f16": f16_bits_to_f64, "bf16": bf16_bits_to_f64}[scale_dtype]
    a = dec(a_h)
    s = dec(s_h)
    b = dec(b_h)
    X = f16_bits_to_f64(X_h).reshape(-1, d_in)
    return forward_factored(U, V, a, s, b, X, rows=rows)


# ---------------------------------------------------------------------------
# Error metric (tolerance reading: row-wise infinity-norm relative error)
# ---------------------------------------------------------------------------

def rowwise_rel_err(y, y_ref) -> float:
    """max over tokens t of max_i |y[t,i] - y_ref[t,i]| / max_i |y_ref[t,i]|.
    A token whose reference row is all zero contributes its absolute error."""
    y = np.asarray(y, dtype=np.float64)
    y_ref = np.asarray(y_ref, dtype=np.float64)
    if y.shape != y_ref.shape:
        raise ValueError(f"shape mismatch {y.shape} vs {y_ref.shape}")
    if y.size == 0:
        return 0.0
    y = y.reshape(-1, y.shape[-1])
    y_ref = y_ref.reshape(-1, y_ref.shape[-1])
    num = np.abs(y - y_ref).max(axis=1)
    den = np.abs(y_ref).max(axis=1)
    den = np.where(den > 0, den, 1.0)
    return float((num / den).max())


# ---------------------------------------------------------------------------
# HiSA budget math (Sec. 3.2 "Hierarchical Shapley Allocation"), as functions
# of given Shapley scores. Plain loops over Python floats.
# ---------------------------------------------------------------------------

def hisa_layer_budgets(phi, B_total: float, tau: float):
    """Eq. hisa_layer_budget: B_l = B_total exp(phi_l / tau) / sum_j exp(phi_j / tau).
    The largest exponent is subtracted first (the ratio is unchanged)."""
    top = max(p / tau for p in phi)
    e = [math.exp(p / tau - top) for p in phi]
    tot = sum(e)
    return [B_total * v / tot for v in e]


def _median(values):
    v = sorted(values)
    k = len(v)
    return v[k // 2] if k % 2 else (v[k // 2 - 1] + v[k // 2]) / 2.0


def mad_z(phi, eps: float):
    """Eq. hisa_mad_norm: (phi_i - median) / (1.4826 MAD + eps), MAD the
    median absolute deviation from the median."""
    med = _median(phi)
    mad = _median([abs(p - med) for p in phi])
    return [(p - med) / (1.4826 * mad + eps) for p in phi]


def hisa_module_budgets(phi_dir, phi_mag, params, B_l: float, alpha: float, eps: float):
    """Module budgets of one layer: MAD z-scores of both distortion scores,
    logistic map P = 1 / (1 + exp(-z)), Soft-OR fusion
    v = 1 - (1 - P_dir)(1 - P_mag), size-aware density
    w = (v / |W| + eps)^alpha and Eq. hisa_module_budget
    b_i = B_l (sum_k |W_k|) w_i / sum_j |W_j| w_j (bits per weight; the
    parameter-weighted mean of the b_i is B_l)."""
    zd, zm = mad_z(phi_dir, eps), mad_z(phi_mag, eps)
    w = []
    for i in range(len(params)):
        pd = 1.0 / (1.0 + math.exp(-zd[i]))
        pm = 1.0 / (1.0 + math.exp(-zm[i]))
        v = 1.0 - (1.0 - pd) * (1.0 - pm)
        w.append((v / params[i] + eps) ** alpha)
    total = float(sum(params))
    den = sum(params[j] * w[j] for j in range(len(params)))
    return [B_l * total * w[i] / den for i in range(len(params))]


def budget_to_rank(b: float, d_out: int, d_in: int, r_max: int = 32768) -> int:
    """App. "Budget-to-rank conversion": r = Round(b d_out d_in / (d_out + d_in))
    (round half up), clipped to [1, r_max]."""
    r = math.floor(b * d_out * d_in / (d_out + d_in) + 0.5)
    return min(max(r, 1), r_max)
