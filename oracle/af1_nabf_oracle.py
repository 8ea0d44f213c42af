"""Plain CPU oracle for NABF, the factorization that produces the AF1 layer
(FP64 numpy).

TEST INFRASTRUCTURE ONLY. Only ``tests/`` and the CPU-baseline leg of
``bench.py`` use it; it shares no code with the CUDA path and does not import
the package.

What it computes: Algorithm NABF (Null-space-Aware Binary Factorization),
Sec. 3.1 and App. "ADMM-SVID Framework in DBF":

    W' = o * W * i^T                       (surrogate, Sec. 3.1)
    W' ~ A B,  A = a * A_pm1 * m1^T (m x r),  B = m2 * B_pm1 * b^T (r x n)

alternating, for t = 1..T,
    left:  A_hat = (W' B^T + rho (A - U_A)) (B B^T + rho I)^-1
           A_q = SVID(A_hat + U_A),  E_A = A_hat - A_q
           P_B = NullProj(B B^T, eta),  A_target = A_hat - E_A P_B
           gamma = ColScaleFit(A_q, A_target),  m1 <- m1 * gamma,  A <- a * A_pm1 * m1^T
    right: B_hat = (A^T A + rho I)^-1 (A^T W' + rho (B - U_B))
           B_q = SVID(B_hat + U_B),  E_B = B_hat - B_q
           P_A = NullProj(A^T A, eta),  B_target = B_hat - P_A E_B
           eta_r = RowScaleFit(B_q, B_target),  m2 <- eta_r * m2,  B <- m2 * B_pm1 * b^T
    duals: U_A <- U_A + A_hat - A,  U_B <- U_B + B_hat - B

Readings where the paper leaves a choice (each also in the design notes):
  * Initialization ("SVID or low-rank approximation"): a randomized range
    finder, A0 = W' Omega with Omega (n x r) of +-1 entries drawn from
    SplitMix64 (seed, index j * r + k), sign = top bit (1 -> -1); then
    B0 = (A0^T A0 + rho I)^-1 A0^T W' (the right proxy with zero prior),
    A = SVID(A0), B = SVID(B0), U_A = U_B = 0.
  * Sign(0) = +1.
  * SVID's rank-1 fit |Z| ~ a m^T: power iteration from the all-ones vector,
    `power_iters` rounds (u = M v / |M v|, v = M^T u, sigma = |v|,
    v = v / sigma); the singular value is split evenly: row scale sqrt(sigma) u,
    column scale sqrt(sigma) v.
  * NullProj(C, eta): eigenvalues lambda_1 >= ... >= lambda_r of the
    symmetric C, k = the first index (0..r) with
    rho_k = sum_{i>k} lambda_i / (sum_i lambda_i + eps) <= eta, and
    P = U_hat U_hat^T over the eigenvectors of lambda_{k+1..r}
    (App. "Adaptive Residual-Energy Cutoff", Eq. app_residual_energy_fraction).
  * ColScaleFit / RowScaleFit: Eq. gamma_solution with eps added to the
    denominator.
  * Duals updated with the compensated factors (A, B after the scale fits).
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
    """NullProj (Sec. 3.1; App. "Adaptive Residual-Energy Cutoff"). Returns
    (P, q) with q = r - k the number of trailing eigenvectors kept."""
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


def nabf(W, r: int, iters: int, rho: float, eta: float = 0.01, eps: float = 1e-8, power_iters: int = 20,
         seed: int = 0, in_scale=None, out_scale=None, compensate: bool = True):
    """Algorithm NABF on W (m x n). Returns dict with U (m x r), V (n x r)
    signs (+-1 int8), a (m), s (r), b (n), the objective history (iters + 1)
    and the number of trailing eigenvectors kept per iteration (left, right)."""
    W = np.asarray(W, dtype=np.float64)
    m, n = W.shape
    i_s = np.ones(n) if in_scale is None else np.asarray(in_scale, dtype=np.float64)
    o_s = np.ones(m) if out_scale is None else np.asarray(out_scale, dtype=np.float64)
    Wp = o_s[:, None] * W * i_s[None, :]
    wn2 = float((Wp * Wp).sum())
    I = np.eye(r)

    Om = splitmix64_signs(seed, n * r).reshape(n, r)
    A0 = Wp @ Om
    B0 = np.linalg.solve(A0.T @ A0 + rho * I, A0.T @ Wp)
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
        # left factor
        CB = B @ B.T
        Ah = np.linalg.solve(CB + rho * I, (Wp @ B.T + rho * (A - UA)).T).T
        Aq, Apm, a, m1 = svid(Ah + UA, power_iters)
        if compensate:
            EA = Ah - Aq
            PB, ql = null_projector(CB, eta, eps)
            At = Ah - EA @ PB
            m1 = m1 * col_scale_fit(Aq, At, eps)
        else:
            ql = 0
        A = a[:, None] * Apm * m1[None, :]
        # right factor
        CA = A.T @ A
        Bh = np.linalg.solve(CA + rho * I, A.T @ Wp + rho * (B - UB))
        Bq, Bpm, m2, b = svid(Bh + UB, power_iters)
        if compensate:
            EB = Bh - Bq
            PA, qr = null_projector(CA, eta, eps)
            Bt = Bh - PA @ EB
            m2 = row_scale_fit(Bq, Bt, eps) * m2
        else:
            qr = 0
        B = m2[:, None] * Bpm * b[None, :]
        # duals
        UA = UA + Ah - A
        UB = UB + Bh - B
        hist.append(objective(A, B))
        q_left.append(ql)
        q_right.append(qr)
    return {"U": Apm.astype(np.int8), "V": Bpm.T.astype(np.int8), "a": a / o_s, "s": m1 * m2, "b": b / i_s,
            "objective": np.array(hist), "q_left": np.array(q_left), "q_right": np.array(q_right),
            "A": A, "B": B, "Wp": Wp}
