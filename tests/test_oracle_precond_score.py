"""Pins for the oracle's Fisher fit, damped inverse, scores and top-k (App. B.2, B.3)."""
import numpy as np
import pytest


def test_fisher_trace_and_symmetry(orc):
    rng = np.random.default_rng(0)
    N, D = 9, 12
    phi = rng.standard_normal((N, D))
    F = orc.fisher(phi)
    np.testing.assert_allclose(F, F.T, rtol=0, atol=0)
    # tr(F) = (1/N) sum_i ||phi_i||^2
    assert abs(np.trace(F) - (phi ** 2).sum() / N) < 1e-12 * np.trace(F)
    np.testing.assert_allclose(F, phi.T @ phi / N, rtol=1e-12)


def test_damping_uses_mean_eigenvalue(orc):
    rng = np.random.default_rng(1)
    D = 10
    Q, _ = np.linalg.qr(rng.standard_normal((D, D)))
    ev = rng.uniform(0.1, 5.0, D)
    F = (Q * ev) @ Q.T
    lam = orc.damping(F, 1e-3, 0.1)
    assert abs(lam - (1e-3 + 0.1 * ev.mean())) < 1e-12


def test_cholesky_matches_library_and_detects_indefinite(orc):
    rng = np.random.default_rng(2)
    X = rng.standard_normal((20, 8))
    M = X.T @ X + 0.5 * np.eye(8)
    L, st = orc.cholesky(M)
    assert st == 0
    np.testing.assert_allclose(L, np.linalg.cholesky(M), rtol=1e-12, atol=1e-12)
    M2 = M.copy()
    M2[5, 5] = -1.0
    _, st2 = orc.cholesky(M2)
    assert st2 > 0


def test_zero_fisher_gives_q_over_lambda(orc):
    D = 6
    Q = np.arange(12, dtype=float).reshape(2, D) - 3
    out = orc.precondition(np.zeros((D, D)), 0.25, Q)
    np.testing.assert_allclose(out, Q / 0.25, rtol=1e-15)


def test_single_example_sherman_morrison(orc):
    # (phi phi^T + lam I)^{-1} q = q/lam - phi (phi.q) / (lam (lam + phi.phi))
    rng = np.random.default_rng(3)
    D, lam = 16, 0.3
    phi = rng.standard_normal(D)
    q = rng.standard_normal((3, D))
    F = orc.fisher(phi[None, :])
    out = orc.precondition(F, lam, q)
    closed = q / lam - np.outer(q @ phi, phi) / (lam * (lam + phi @ phi))
    np.testing.assert_allclose(out, closed, rtol=1e-11, atol=1e-12)


def test_preconditioned_residual_is_small(orc):
    rng = np.random.default_rng(4)
    N, D = 30, 20
    phi = rng.standard_normal((N, D))
    F = orc.fisher(phi)
    lam = orc.damping(F, 0.0, 1e-2)
    Q = rng.standard_normal((5, D))
    X = orc.precondition(F, lam, Q)
    R = X @ (F + lam * np.eye(D)) - Q
    assert np.abs(R).max() < 1e-12 * np.abs(Q).max() * 100


def test_score_is_the_inner_product(orc):
    rng = np.random.default_rng(5)
    Qh = rng.standard_normal((4, 33))
    phi = rng.standard_normal((7, 33))
    np.testing.assert_allclose(orc.score(Qh, phi), Qh @ phi.T, rtol=1e-13)


def test_topk_matches_brute_force_with_ties(orc):
    rng = np.random.default_rng(6)
    S = np.round(rng.standard_normal((5, 200)) * 4) / 4  # many exact ties
    k = 37
    idx, val = orc.topk(S, k)
    for q in range(S.shape[0]):
        order = sorted(range(S.shape[1]), key=lambda i: (-S[q, i], i))[:k]
        assert list(idx[q]) == order
        np.testing.assert_array_equal(val[q], S[q, order])


@pytest.mark.parametrize("k", [1, 100])
def test_topk_full_row_when_k_equals_n(orc, k):
    S = np.linspace(-1, 1, k)[None, :]
    idx, _ = orc.topk(S, k)
    assert list(idx[0]) == list(range(k - 1, -1, -1))


def test_fisher_entry_is_the_ordered_sum_over_examples(orc):
    # F[a][b] = (sum over n in order of phi_na phi_nb) / N, bit for bit
    rng = np.random.default_rng(7)
    N, D = 11, 5
    phi = rng.standard_normal((N, D))
    F = orc.fisher(phi)
    for a in range(D):
        for b in range(D):
            s = 0.0
            for n in range(N):
                s += phi[n, a] * phi[n, b]
            assert F[a, b] == s / N


def test_damping_from_features_equals_damping_of_fisher(orc):
    rng = np.random.default_rng(8)
    phi = rng.standard_normal((13, 9))
    assert orc.damping_features(phi, 1e-3, 1e-2) == orc.damping(orc.fisher(phi), 1e-3, 1e-2)


@pytest.mark.parametrize("N,D", [(6, 40), (40, 12), (1, 7)])
def test_lowrank_precondition_agrees_with_cholesky_route(orc, N, D):
    # Woodbury (N x N solve) and the D x D Cholesky solve of the same (F + lambda I)
    rng = np.random.default_rng(N * 100 + D)
    phi = rng.standard_normal((N, D)) * rng.uniform(0.5, 2.0, D)
    Q = rng.standard_normal((4, D))
    F = orc.fisher(phi)
    lam = orc.damping(F, 0.0, 1e-2)
    a = orc.precondition_lowrank(phi, lam, Q)
    b = orc.precondition(F, lam, Q)
    np.testing.assert_allclose(a, b, rtol=1e-9, atol=1e-12 * np.abs(b).max())
    c = np.linalg.solve(phi.T @ phi / N + lam * np.eye(D), Q.T).T
    np.testing.assert_allclose(a, c, rtol=1e-9, atol=1e-12 * np.abs(c).max())


def test_topk_nan_ranks_first_and_signed_zeros_tie(orc):
    # NaN is ranked above +inf (NaNs among themselves by index); -0 and +0 are equal
    S = np.array([[0.0, np.nan, -0.0, 1.0, np.inf, np.nan, -np.inf, 0.0, -1.0]])
    idx, val = orc.topk(S, 9)
    assert list(idx[0]) == [1, 5, 4, 3, 0, 2, 7, 8, 6]
    assert np.isnan(val[0, :2]).all() and list(val[0, 2:4]) == [np.inf, 1.0]
