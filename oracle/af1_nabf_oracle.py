"""Plain CPU oracle for NABF, the factorization that produces the AF1 layer
(FP64 numpy).

TEST INFRASTRUCTURE ONLY. Only ``tests/`` and the CPU-baseline leg of
``bench.py`` use it; it shares no code with the CUDA path and does not import
the package.

What it computes: the NABF factorization (Null-space-Aware Binary
Factorization) of Sec. 3.1 and App. "ADMM-SVID Framework in DBF". The
weight, reweighted by the surrogate's output and input statistics
(W' = o * W * i^T), is approximated by A B with A = a * A_pm1 * m1^T (m x r)
and B = m2 * B_pm1 * b^T (r x n): binary sign matrices with rank-1 magnitude
scales. Each iteration updates the left factor, then the right one, each by
one step of scaled ADMM on the constrained least-squares problem
min ||W' - A B||_F^2 (the other factor held fixed):

  * proxy: the unconstrained regularised least-squares solution around the
    current factor minus its scaled dual (App. "Closed-form proxy updates",
    App. "ADMM subproblem"); left_proxy / right_proxy;
  * projection: SVID of proxy + dual (signs and a rank-1 magnitude fit);
  * null-space compensation (Sec. 3.1): the projection residual is removed
    along the directions the other factor cannot see (the trailing
    eigenvectors of its Gram matrix, cut off by residual energy, App.
    "Adaptive Residual-Energy Cutoff"), and the per-rank magnitude of the
    binary factor is refitted to that target in closed form (Eq.
    gamma_solution); compensated_scale;
  * dual step: dual + proxy - factor (dual_step).

Readings where the paper leaves a choice (each also in the design notes):
  * Initialization: a randomized range finder, A0 = W' Omega with Omega
    (n x r) of +-1 entries drawn from SplitMix64 (seed, index j * r + k),
    sign = top bit (1 -> -1); then B0 = the right proxy with a zero prior,
    A = SVID(A0), B = SVID(B0), both duals zero.
  * Sign(0) = +1.
  * SVID's rank-1 fit |Z| ~ a m^T: power iteration from the all-ones vector,
    `power_iters` rounds (u = M v / |M v|, v = M^T u, sigma = |v|,
    v = v / sigma); the singular value is split evenly: row scale sqrt(sigma) u,
    column scale sqrt(sigma) v.
  * Null-space projector of a symmetric Gram matrix C: eigenvalues
    lambda_1 >= ... >= lambda_r, k = the first index (0..r) with
    rho_k = sum_{i>k} lambda_i / (sum_i lambda_i + eps) <= eta, and
    P = U_hat U_hat^T over the eigenvectors of lambda_{k+1..r}
    (Eq. app_residual_energy_fraction).
  * Scale fits: Eq. gamma_solution with eps added to the denominator.
  * Duals updated with the compensated factors (after the scale fits).
  * Output in AF1 form: U = A_pm1, V = B_pm1^T, s = m1 * m2, and the
    surrogate undone in the outer scales: a <- a / o, b <- b / i.
  * Objective: |W' - A B|_F^2 / |W'|_F^2 after the initialization and after
    every iteration.
"""
import numpy as np

_M64 = (1 << 64) - 1


def splitmix64(seed: int, count: int) -> np.ndarray:
    """SplitMix64 outputs for indices 0..count-1 (uint64): z = seed + (idx + 1)
    * 0x9E3779B97F4A7C15, then the published mixing steps (Steele, Lea and
    Flood, 2014)."""
    idx = np.arange(1, count + 1, dtype=np.uint64)
    with np.errstate(over="ignore"):
        z = np.uint64(seed & _M64) + idx * np.uint64(0x9E3779B97F4A7C15)
        z = (z ^ (z >> np.uint64(30))) * np.uint64(0xBF58476D1CE4E5B9)
        z = (z ^ (z >> np.uint64(27))) * np.uint64(0x94D049BB133111EB)
        z = z ^ (z >> np.uint64(31))
    return z


def splitmix64_signs(seed: int, count: int) -> np.ndarray:
    """+-1 (float64) for indices 0..count-1: top bit of SplitMix64 set -> -1."""
    return np.where((splitmix64(seed, count) >> np.uint64(63)) != 0, -1.0, 1.0)


def sign_pm1(Z) -> np.ndarray:
    """Sign with Sign(0) = +1."""
    return np.where(np.asarray(Z) < 0, -1.0, 1.0)


def svid(Z, power_iters: int):
    """SVID projection (App. "SVID projection"): signs of Z and a rank-1 fit of
    |Z| by power iteration. Returns (Zq, signs, row_scale, col_scale)."""
    Z = np.asarray(Z, dtype=np.float64)
    S = sign_pm1(Z)
    M = np.abs(Z)
    v = np.ones(M.shape[1]) / np.sqrt(M.shape[1])
    sigma = 0.0
    for _ in range(max(power_iters, 1)):
        u = M @ v
        nu = np.linalg.norm(u)
        u = u / nu if nu > 0 else u
        v = M.T @ u
        sigma = np.linalg.norm(v)
        v = v / sigma if sigma > 0 else v
    rs = np.sqrt(sigma) * u
    cs = np.sqrt(sigma) * v
    return rs[:, None] * S * cs[None, :], S, rs, cs


def null_projector(C, eta: float, eps: float):
    """Projector onto the trailing eigenvectors of the symmetric Gram matrix C
    that hold at most a fraction eta of its energy (Sec. 3.1; App.
    "Adaptive Residual-Energy Cutoff"). Returns (P, q) with q = r - k the
    number of trailing eigenvectors kept."""
    C = np.asarray(C, dtype=np.float64)
    lam, Q = np.linalg.eigh(0.5 * (C + C.T))      # ascending
    lam = lam[::-1]                                # descending
    Q = Q[:, ::-1]
    total = lam.sum()
    r = lam.shape[0]
    k = r
    for kk in range(r + 1):
        if lam[kk:].sum() / (total + eps) <= eta:
            k = kk
            break
    Uh = Q[:, k:]
    return Uh @ Uh.T, r - k


def col_scale_fit(Aq, At, eps: float) -> np.ndarray:
    """gamma* = diag(Aq^T At) / (diag(Aq^T Aq) + eps)  (Eq. gamma_solution)."""
    return np.einsum("ij,ij->j", Aq, At) / (np.einsum("ij,ij->j", Aq, Aq) + eps)


def row_scale_fit(Bq, Bt, eps: float) -> np.ndarray:
    """The symmetric fit over the rows of the right factor."""
    return np.einsum("ij,ij->i", Bq, Bt) / (np.einsum("ij,ij->i", Bq, Bq) + eps)


def left_proxy(Wp, B, A, UA, rho: float):
    """argmin_X |W' - X B|_F^2 + rho |X - (A - UA)|_F^2
    = (W' B^T + rho (A - UA)) (B B^T + rho I)^-1."""
    r = B.shape[0]
    return np.linalg.solve(B @ B.T + rho * np.eye(r), (Wp @ B.T + rho * (A - UA)).T).T


def right_proxy(Wp, A, B, UB, rho: float):
    """argmin_Y |W' - A Y|_F^2 + rho |Y - (B - UB)|_F^2
    = (A^T A + rho I)^-1 (A^T W' + rho (B - UB))."""
    r = A.shape[1]
    return np.linalg.solve(A.T @ A + rho * np.eye(r), A.T @ Wp + rho * (B - UB))


def compensated_scale(Zq, Zh, P, side: str, eps: float) -> np.ndarray:
    """Null-space compensation (Sec. 3.1) and the closed-form magnitude refit
    (Eq. gamma_solution): the projection residual Zh - Zq is removed along the
    projector P (acting on the rank index: from the right for the left
    factor, from the left for the right factor), and the per-rank scale that
    best maps Zq onto that target is returned."""
    R = Zh - Zq
    if side == "left":
        return col_scale_fit(Zq, Zh - R @ P, eps)
    return row_scale_fit(Zq, Zh - P @ R, eps)


def dual_step(U, proxy, factor):
    """Scaled dual update: U + proxy - factor."""
    return U + proxy - factor


def nabf(W, r: int, iters: int, rho: float, eta: float = 0.01, eps: float = 1e-8, power_iters: int = 20,
         seed: int = 0, in_scale=None, out_scale=None, compensate: bool = True):
    """NABF (Algorithm NABF) on W (m x n). Returns dict with U (m x r), V (n x r)
    signs (+-1 int8), a (m), s (r), b (n), the objective history (iters + 1)
    and the number of trailing eigenvectors kept per iteration (left, right)."""
    W = np.asarray(W, dtype=np.float64)
    m, n = W.shape
    i_s = np.ones(n) if in_scale is None else np.asarray(in_scale, dtype=np.float64)
    o_s = np.ones(m) if out_scale is None else np.asarray(out_scale, dtype=np.float64)
    Wp = o_s[:, None] * W * i_s[None, :]
    wn2 = float((Wp * Wp).sum())
    Om = splitmix64_signs(seed, n * r).reshape(n, r)
    A0 = Wp @ Om
    B0 = right_proxy(Wp, A0, np.zeros((r, n)), np.zeros((r, n)), rho)
    A, Apm, a, m1 = svid(A0, power_iters)
    B, Bpm, m2, b = svid(B0, power_iters)
    UA = np.zeros_like(A)
    UB = np.zeros_like(B)

    def objective(A, B):
        D = Wp - A @ B
        return float((D * D).sum()) / wn2

    hist = [objective(A, B)]
    q_left, q_right = [0], [0]
    for _ in range(iters):
        # left factor: proxy, projection, compensated magnitudes
        Ah = left_proxy(Wp, B, A, UA, rho)
        Aq, Apm, a, m1 = svid(Ah + UA, power_iters)
        ql = 0
        if compensate:
            PB, ql = null_projector(B @ B.T, eta, eps)
            m1 = m1 * compensated_scale(Aq, Ah, PB, "left", eps)
        A = a[:, None] * Apm * m1[None, :]
        # right factor, against the new left factor
        Bh = right_proxy(Wp, A, B, UB, rho)
        Bq, Bpm, m2, b = svid(Bh + UB, power_iters)
        qr = 0
        if compensate:
            PA, qr = null_projector(A.T @ A, eta, eps)
            m2 = compensated_scale(Bq, Bh, PA, "right", eps) * m2
        B = m2[:, None] * Bpm * b[None, :]
        UA = dual_step(UA, Ah, A)
        UB = dual_step(UB, Bh, B)
        hist.append(objective(A, B))
        q_left.append(ql)
        q_right.append(qr)
    return {"U": Apm.astype(np.int8), "V": Bpm.T.astype(np.int8), "a": a / o_s, "s": m1 * m2, "b": b / i_s,
            "objective": np.array(hist), "q_left": np.array(q_left), "q_right": np.array(q_right),
            "A": A, "B": B, "Wp": Wp}
