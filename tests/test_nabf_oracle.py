"""Pins of the NABF oracle (Algorithm NABF; App. "ADMM-SVID Framework in
DBF", "Adaptive Residual-Energy Cutoff"): each step against what the
mathematics fixes independently of the code."""
import numpy as np
import pytest

from oracle import af1_nabf_oracle as N


def test_splitmix64_published_outputs():
    # The generator's first outputs from state 0 (its reference sequence).
    z = N.splitmix64(0, 4)
    assert [int(v) for v in z] == [0xE220A8397B1DCDAF, 0x6E789E6AA1B965F4, 0x06C45D188009454F, 0xF88BB8A8724C81EC]
    np.testing.assert_array_equal(N.splitmix64_signs(0, 4), [-1.0, 1.0, 1.0, -1.0])


def test_svid_reproduces_a_signed_rank_one_magnitude():
    g = np.random.default_rng(0)
    x, y = g.uniform(0.5, 2.0, 40), g.uniform(0.1, 3.0, 25)
    S = np.where(g.random((40, 25)) < 0.5, -1.0, 1.0)
    Z = S * np.outer(x, y)
    Zq, Sq, rs, cs = N.svid(Z, 3)
    np.testing.assert_allclose(Zq, Z, rtol=1e-12)
    np.testing.assert_array_equal(Sq, S)
    np.testing.assert_allclose(np.outer(rs, cs), np.outer(x, y), rtol=1e-12)


def test_svid_magnitude_is_the_top_singular_pair():
    g = np.random.default_rng(1)
    Z = g.normal(size=(30, 20))
    _, S, rs, cs = N.svid(Z, 200)
    U, sv, Vt = np.linalg.svd(np.abs(Z))
    np.testing.assert_allclose(np.outer(rs, cs), sv[0] * np.outer(np.abs(U[:, 0]), np.abs(Vt[0])), rtol=1e-9)
    np.testing.assert_array_equal(S, np.where(Z < 0, -1.0, 1.0))
    assert N.sign_pm1(np.array([0.0, -0.0]))[0] == 1.0


def test_null_projector_energy_cutoff():
    g = np.random.default_rng(2)
    Q, _ = np.linalg.qr(g.normal(size=(5, 5)))
    lam = np.array([100.0, 50.0, 1.0, 0.5, 0.0])
    C = Q @ np.diag(lam) @ Q.T
    # rho_1 = 51.5 / 151.5 > 0.01, rho_2 = 1.5 / 151.5 = 0.0099 <= 0.01: keep 3 trailing vectors
    P, q = N.null_projector(C, 0.01, 1e-12)
    assert q == 3
    np.testing.assert_allclose(P, Q[:, 2:] @ Q[:, 2:].T, atol=1e-12)
    np.testing.assert_allclose(P @ P, P, atol=1e-12)
    # A factor B with B B^T = C: |P B|^2 / |B|^2 is the residual-energy fraction.
    R, _ = np.linalg.qr(g.normal(size=(9, 5)))
    B = Q @ np.diag(np.sqrt(lam)) @ R.T
    frac = np.linalg.norm(P @ B) ** 2 / np.linalg.norm(B) ** 2
    assert frac == pytest.approx(1.5 / 151.5, rel=1e-10)
    # Scale invariance of the cutoff.
    _, q2 = N.null_projector(1e6 * C, 0.01, 1e-12)
    assert q2 == 3
    # eta below the smallest nonzero fraction keeps only the zero direction.
    _, q3 = N.null_projector(C, 0.001, 1e-12)
    assert q3 == 1


def test_scale_fits_are_least_squares_optima():
    g = np.random.default_rng(3)
    Aq = g.normal(size=(50, 8))
    c = g.uniform(0.5, 2.0, 8)
    np.testing.assert_allclose(N.col_scale_fit(Aq, Aq * c[None, :], 0.0), c, rtol=1e-12)
    At = Aq * c[None, :] + 0.3 * g.normal(size=(50, 8))
    gam = N.col_scale_fit(Aq, At, 0.0)
    f = lambda v: np.sum((At - Aq * v[None, :]) ** 2)
    for j in range(8):
        for d in (1e-4, -1e-4):
            v = gam.copy()
            v[j] += d
            assert f(v) > f(gam)
    Bq = g.normal(size=(6, 40))
    Bt = c[:6, None] * Bq
    np.testing.assert_allclose(N.row_scale_fit(Bq, Bt, 0.0), c[:6], rtol=1e-12)


def test_nabf_output_maps_back_to_the_factors():
    g = np.random.default_rng(4)
    m, n, r = 48, 40, 12
    W = g.normal(size=(m, n))
    i_s, o_s = g.uniform(0.5, 2.0, n), g.uniform(0.5, 2.0, m)
    out = N.nabf(W, r, iters=4, rho=1.0, in_scale=i_s, out_scale=o_s, seed=7)
    U, V = out["U"].astype(np.float64), out["V"].astype(np.float64)
    W_hat = out["a"][:, None] * (U * out["s"][None, :]) @ V.T * out["b"][None, :]
    # The AF1 layer is A B with the surrogate scaling undone.
    np.testing.assert_allclose(W_hat, out["A"] @ out["B"] / np.outer(o_s, i_s), rtol=1e-10, atol=1e-12)
    assert set(np.unique(U)) <= {-1.0, 1.0} and set(np.unique(V)) <= {-1.0, 1.0}
    np.testing.assert_allclose(out["Wp"], o_s[:, None] * W * i_s[None, :])
    assert np.all(np.isfinite(out["objective"])) and out["objective"].shape == (5,)


def test_nabf_improves_on_its_initialisation_and_dbf_has_no_projector():
    g = np.random.default_rng(5)
    m, n, r = 64, 48, 16
    W = g.normal(size=(m, r)) @ g.normal(size=(r, n)) + 0.1 * g.normal(size=(m, n))
    for comp in (True, False):
        out = N.nabf(W, r, iters=8, rho=1.0, compensate=comp)
        assert out["objective"][-1] < out["objective"][0]
        assert (np.all(out["q_left"] == 0) and np.all(out["q_right"] == 0)) == (not comp)


def test_proxies_satisfy_first_order_optimality(monkeypatch):
    """The ADMM proxies (Sec. 3.1) are regularised least-squares minimisers:
    the gradient of |W' - A0 B|^2 + rho |B|^2 vanishes at the initial right
    proxy B0, and that of |W' - A B|^2 + rho |A - A_prev|^2 at the first left
    proxy (duals still zero), A_prev and B being the SVID projections of the
    initialisation. The initial sketch is W' times the SplitMix64 signs."""
    g = np.random.default_rng(6)
    m, n, r, rho = 30, 24, 6, 0.7
    W = g.normal(size=(m, n))
    calls = []
    real = N.svid

    def spy(Z, power_iters):
        out = real(Z, power_iters)
        calls.append((np.array(Z, dtype=np.float64), out))
        return out

    monkeypatch.setattr(N, "svid", spy)
    N.nabf(W, r, iters=1, rho=rho, seed=3)
    assert len(calls) == 4  # init A, init B, then the left and right projections of iteration 1
    (A0, (A_init, *_)), (B0, (B_init, *_)), (Ah, _) = calls[0], calls[1], calls[2]
    np.testing.assert_allclose(A0, W @ N.splitmix64_signs(3, n * r).reshape(n, r), rtol=1e-12, atol=1e-12)
    grad_B = -A0.T @ (W - A0 @ B0) + rho * B0
    assert np.abs(grad_B).max() <= 1e-9 * np.abs(A0.T @ W).max()
    grad_A = -(W - Ah @ B_init) @ B_init.T + rho * (Ah - A_init)
    assert np.abs(grad_A).max() <= 1e-9 * np.abs(W @ B_init.T).max()
    # A transposed operand or a dropped regulariser fails the same check.
    wrong = np.linalg.solve(B_init @ B_init.T, (W @ B_init.T).T).T
    assert np.abs(-(W - wrong @ B_init) @ B_init.T + rho * (wrong - A_init)).max() > 1e-3


def _admm_left(Wp, B, rho, project, dual, iters):
    """The oracle's left-factor ADMM step (proxy, projection of proxy + dual,
    dual step) iterated with B held fixed."""
    m, r = Wp.shape[0], B.shape[0]
    A = np.zeros((m, r))
    U = np.zeros_like(A)
    with np.errstate(all="ignore"):
        for _ in range(iters):
            Ah = N.left_proxy(Wp, B, A, U, rho)
            A = project(Ah + U)
            U = dual(U, Ah, A)
    return A


def test_dual_update_pinned_by_a_convex_constraint():
    """Scaled ADMM converges to the constrained least-squares minimiser when
    the projection is onto a convex set (App. "ADMM subproblem"). Take the
    set of m x r matrices whose columns S are zero: its Euclidean projection
    zeroes those columns and min |W' - A B|^2 over it has the closed form
    A_free = W' B_free^T (B_free B_free^T)^-1, A_S = 0. B is not orthonormal,
    so without the dual (or with its sign flipped) the iteration ends
    elsewhere: both mutants are rejected."""
    g = np.random.default_rng(5)
    m, n, r = 12, 30, 6
    Wp = g.normal(size=(m, n))
    B = g.normal(size=(r, r)) @ g.normal(size=(r, n)) / 3  # correlated rows
    S = [1, 4]
    free = [j for j in range(r) if j not in S]

    def project(Z):
        Z = Z.copy()
        Z[:, S] = 0.0
        return Z

    Bf = B[free]
    A_star = np.zeros((m, r))
    A_star[:, free] = Wp @ Bf.T @ np.linalg.inv(Bf @ Bf.T)
    A = _admm_left(Wp, B, 3.0, project, N.dual_step, 400)
    np.testing.assert_allclose(A, A_star, atol=1e-9)
    flipped = _admm_left(Wp, B, 3.0, project, lambda U, P, F: U - P + F, 400)
    dropped = _admm_left(Wp, B, 3.0, project, lambda U, P, F: U, 400)
    for bad in (flipped, dropped):
        assert not np.all(np.isfinite(bad)) or np.abs(bad - A_star).max() > 1e-2
