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
