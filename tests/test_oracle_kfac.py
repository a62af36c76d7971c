"""Pins for the oracle's Kronecker-factored curvature on projected factors
(K-FAC, EK-FAC; applied to projected factors per App. A.2, damped by a multiple
of the mean eigenvalue per App. B.2)."""
import numpy as np
import pytest


def _spd(rng, n, spread=1.0):
    X = rng.standard_normal((n, n))
    return X @ X.T / n + spread * np.diag(rng.uniform(0.1, 1.0, n))


@pytest.mark.parametrize("n", [1, 2, 7, 32, 64])
def test_jacobi_matches_lapack(orc, n):
    rng = np.random.default_rng(n)
    C = _spd(rng, n)
    w, U, sweeps = orc.sym_eig(C)
    assert 0 <= sweeps <= 20
    np.testing.assert_allclose(w, np.linalg.eigvalsh(C), rtol=1e-12, atol=1e-13 * np.abs(w).max())
    np.testing.assert_allclose(U.T @ U, np.eye(n), atol=1e-13)
    np.testing.assert_allclose(U @ np.diag(w) @ U.T, C, atol=1e-13 * np.abs(C).max())


def test_jacobi_two_by_two_closed_form_and_diagonal(orc):
    a, b, d = 3.0, -1.25, 0.5
    w, U, _ = orc.sym_eig(np.array([[a, b], [b, d]]))
    m, r = (a + d) / 2, np.hypot((a - d) / 2, b)
    np.testing.assert_allclose(w, [m - r, m + r], rtol=1e-15)
    D = np.diag([4.0, -1.0, 2.0])
    w, U, sweeps = orc.sym_eig(D)
    assert sweeps == 0
    np.testing.assert_array_equal(w, [-1.0, 2.0, 4.0])
    np.testing.assert_array_equal(np.abs(U), np.eye(3)[:, [1, 2, 0]])


def test_covariances_brute_force_and_identity_map(orc):
    rng = np.random.default_rng(1)
    N, T, di, do, ki, ko = 3, 5, 12, 8, 4, 6
    A, B = rng.standard_normal((N, T, di)), rng.standard_normal((N, T, do))
    Ca, Cg = orc.kfac_covariances(A, B, ki, ko, seed=2, layer=3)
    P_in, P_out = orc.proj_matrix(2, 3, 0, di, ki), orc.proj_matrix(2, 3, 1, do, ko)
    At, Bt = (A @ P_in).reshape(-1, ki), (B @ P_out).reshape(-1, ko)
    np.testing.assert_allclose(Ca, At.T @ At / (N * T), rtol=1e-12)
    np.testing.assert_allclose(Cg, Bt.T @ Bt / (N * T), rtol=1e-12)
    Ca, Cg = orc.kfac_covariances(A, B, di, do, seed=0, layer=0, kind=1)
    Af, Bf = A.reshape(-1, di), B.reshape(-1, do)
    np.testing.assert_allclose(Ca, Af.T @ Af / (N * T), rtol=1e-12)
    np.testing.assert_allclose(Cg, Bf.T @ Bf / (N * T), rtol=1e-12)


def _basis(orc, rng, ki, ko):
    wa, Ua, _ = orc.sym_eig(_spd(rng, ki))
    wg, Ug, _ = orc.sym_eig(_spd(rng, ko))
    return wa, Ua, wg, Ug


def test_kfac_precondition_is_the_damped_kronecker_inverse(orc):
    # (Cg (x) Ca + lambda I)^{-1} q by a dense solve, features indexed r*k_in + c
    rng = np.random.default_rng(2)
    ki, ko, nq = 5, 3, 4
    Ca, Cg = _spd(rng, ki), _spd(rng, ko)
    wa, Ua, _ = orc.sym_eig(Ca)
    wg, Ug, _ = orc.sym_eig(Cg)
    Lam = orc.kfac_eigenvalues(wa, wg)
    lam = orc.kfac_damping(Lam, 0.0, 0.1)
    np.testing.assert_allclose(lam, 0.1 * np.trace(Ca) * np.trace(Cg) / (ki * ko), rtol=1e-13)
    Q = rng.standard_normal((nq, ko * ki))
    Qh = orc.kfac_precondition(Ua, Ug, Lam, lam, Q)
    K = np.kron(Cg, Ca) + lam * np.eye(ki * ko)
    np.testing.assert_allclose(Qh, np.linalg.solve(K, Q.T).T, rtol=1e-11, atol=1e-13)


def test_ekfac_eigenvalues_are_the_fisher_diagonal_in_the_kronecker_basis(orc):
    # EK-FAC's correction is diag(U^T F U) with U = Ug (x) Ua and F the empirical Fisher;
    # its eigenvalues sum to tr(F); its preconditioner is (U diag(Lam) U^T + lambda I)^{-1}
    rng = np.random.default_rng(3)
    ki, ko, N = 4, 6, 9
    wa, Ua, wg, Ug = _basis(orc, rng, ki, ko)
    phi = rng.standard_normal((N, ko, ki)) * rng.uniform(0.5, 2.0, (N, 1, 1))
    Lam = orc.ekfac_eigenvalues(phi, Ua, Ug)
    F = orc.fisher(phi)
    U = np.kron(Ug, Ua)
    np.testing.assert_allclose(Lam.reshape(-1), np.diag(U.T @ F @ U), rtol=1e-12)
    np.testing.assert_allclose(Lam.sum(), np.trace(F), rtol=1e-12)
    lam = orc.kfac_damping(Lam, 1e-3, 0.1)
    Q = rng.standard_normal((3, ki * ko))
    Qh = orc.kfac_precondition(Ua, Ug, Lam, lam, Q)
    K = U @ np.diag(Lam.reshape(-1)) @ U.T + lam * np.eye(ki * ko)
    np.testing.assert_allclose(Qh, np.linalg.solve(K, Q.T).T, rtol=1e-11, atol=1e-13)


def test_ekfac_is_exact_when_the_fisher_is_diagonal_in_the_basis(orc):
    # features that are scaled basis vectors u_g[r] u_a[c]^T: F is then diagonal in
    # the Kronecker basis and EK-FAC's preconditioner equals the exact (F + lambda I)^{-1}
    rng = np.random.default_rng(4)
    ki, ko = 3, 2
    _, Ua, _, Ug = _basis(orc, rng, ki, ko)
    phi = np.stack([s * np.outer(Ug[:, r], Ua[:, c]) for r in range(ko) for c in range(ki)
                    for s in (1.5 + r + c, -(0.5 + c))])
    Lam = orc.ekfac_eigenvalues(phi, Ua, Ug)
    F = orc.fisher(phi)
    Q = rng.standard_normal((2, ki * ko))
    Qh = orc.kfac_precondition(Ua, Ug, Lam, 0.01, Q)
    np.testing.assert_allclose(Qh, orc.precondition(F, 0.01, Q), rtol=1e-10)
