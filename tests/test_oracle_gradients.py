"""Pins for the oracle's gradients, projections and similarities (Eq. 1, Eq. 2, Eq. 4)."""
import itertools

import numpy as np
import pytest


def _rand(rng, *shape, scale=1.0):
    return rng.standard_normal(shape) * scale


def test_materialize_matches_finite_difference_of_a_linear_layer(orc):
    # l(W) = 1/2 sum_t ||W a_t - y_t||^2 has dl/dW = sum_t g_t a_t^T with
    # g_t = W a_t - y_t (the chain rule of Sec. 3.2). l is quadratic in W, so
    # the central difference is exact up to rounding.
    rng = np.random.default_rng(0)
    T, d_in, d_out = 5, 4, 3
    A = _rand(rng, T, d_in)          # rows a_t
    Y = _rand(rng, T, d_out)
    W = _rand(rng, d_out, d_in)

    def loss(Wm):
        R = A @ Wm.T - Y
        return 0.5 * float((R * R).sum())

    Bg = A @ W.T - Y                 # rows g_t = W a_t - y_t
    G = orc.materialize(A, Bg)
    h = 1e-3
    fd = np.empty_like(W)
    for r in range(d_out):
        for c in range(d_in):
            E = np.zeros_like(W)
            E[r, c] = h
            fd[r, c] = (loss(W + E) - loss(W - E)) / (2 * h)
    assert G.shape == (d_out, d_in)
    np.testing.assert_allclose(G, fd, rtol=1e-8, atol=1e-9)


def test_materialize_is_sum_of_token_outer_products(orc):
    rng = np.random.default_rng(1)
    T, d_in, d_out = 7, 5, 6
    A, B = _rand(rng, T, d_in), _rand(rng, T, d_out)
    brute = sum(np.outer(B[t], A[t]) for t in range(T))
    np.testing.assert_allclose(orc.materialize(A, B), brute, rtol=1e-13, atol=1e-13)


def test_factor_projection_is_the_kronecker_map_of_vec(orc):
    # Eq. 2: sum_t a~_t (x) g~_t = (P_a (x) P_g) vec(DW), vec stacking columns.
    rng = np.random.default_rng(2)
    T, d_in, d_out, k_in, k_out = 6, 5, 4, 3, 2
    A, B = _rand(rng, T, d_in), _rand(rng, T, d_out)
    P_in = orc.proj_matrix(9, 1, 0, d_in, k_in)    # = P_a^T
    P_out = orc.proj_matrix(9, 1, 1, d_out, k_out)  # = P_g^T
    phi = orc.project_with(A, B, P_in, P_out)       # k_out x k_in
    gamma = orc.materialize(A, B).flatten(order="F")
    kron = np.kron(P_in.T, P_out.T) @ gamma         # length k_in*k_out, column-stacked
    np.testing.assert_allclose(phi.flatten(order="F"), kron, rtol=1e-12, atol=1e-12)


@pytest.mark.parametrize("shape", [(1, 3, 8, 6, 4, 2), (3, 9, 16, 24, 8, 4), (2, 1, 64, 32, 16, 16)])
def test_factored_and_materialized_routes_agree(orc, shape):
    N, T, d_in, d_out, k_in, k_out = shape
    rng = np.random.default_rng(3)
    A, B = _rand(rng, N, T, d_in), _rand(rng, N, T, d_out, scale=0.1)
    pa = orc.project(A, B, k_in, k_out, seed=0, layer=2, route="factored")
    pb = orc.project(A, B, k_in, k_out, seed=0, layer=2, route="materialized")
    np.testing.assert_allclose(pa, pb, rtol=1e-11, atol=1e-12 * np.abs(pa).max())


def test_identity_projection_reproduces_the_gradient(orc):
    rng = np.random.default_rng(4)
    N, T, d = 3, 5, 8
    A, B = _rand(rng, N, T, d), _rand(rng, N, T, d)
    phi = orc.project(A, B, d, d, seed=1, layer=0, kind=1)
    for n in range(N):
        np.testing.assert_allclose(phi[n], orc.materialize(A[n], B[n]), rtol=1e-13, atol=1e-13)


@pytest.mark.parametrize("k_in,k_out", [(1, 1), (1, 2), (2, 1), (2, 2)])
def test_projection_preserves_norm_in_expectation_exact_enumeration(orc, k_in, k_out):
    # E ||(P_a (x) P_g) gamma||^2 = ||gamma||^2 for entries +-1/sqrt(k) (App. A.2):
    # average over every sign pattern of both maps at d_in = d_out = 2.
    rng = np.random.default_rng(5)
    T, d = 3, 2
    A, B = _rand(rng, T, d), _rand(rng, T, d)
    g2 = float((orc.materialize(A, B) ** 2).sum())
    total, count = 0.0, 0
    for si in itertools.product((-1.0, 1.0), repeat=d * k_in):
        P_in = np.array(si).reshape(d, k_in) / np.sqrt(k_in)
        for so in itertools.product((-1.0, 1.0), repeat=d * k_out):
            P_out = np.array(so).reshape(d, k_out) / np.sqrt(k_out)
            total += float((orc.project_with(A, B, P_in, P_out) ** 2).sum())
            count += 1
    assert abs(total / count - g2) < 1e-12 * g2


def test_projection_preserves_norm_in_expectation_over_seeds(orc):
    # Monte Carlo over 1000 seeds of the hashed maps at a 256x256 layer, T = 32, k = 16.
    rng = np.random.default_rng(6)
    T, d, k = 32, 256, 16
    A, B = _rand(rng, 1, T, d), _rand(rng, 1, T, d, scale=0.1)
    g2 = float((orc.materialize(A[0], B[0]) ** 2).sum())
    ratios = np.array([float((orc.project(A, B, k, k, seed=s, layer=0) ** 2).sum()) / g2
                       for s in range(1000)])
    se = ratios.std(ddof=1) / np.sqrt(ratios.size)
    assert abs(ratios.mean() - 1.0) < 4 * se


def test_gram_identity_equals_materialized_frobenius(orc):
    # Eq. 4 against <DW_q, DW_i>_F from Eq. 1
    rng = np.random.default_rng(7)
    T, d_in, d_out = 6, 7, 5
    Aq, Bq = _rand(rng, 2, T, d_in), _rand(rng, 2, T, d_out)
    At, Bt = _rand(rng, 3, T, d_in), _rand(rng, 3, T, d_out)
    Sg = orc.similarity(Aq, Bq, At, Bt, route="gram")
    Sm = orc.similarity(Aq, Bq, At, Bt, route="materialized")
    brute = np.array([[float((orc.materialize(Aq[q], Bq[q]) * orc.materialize(At[i], Bt[i])).sum())
                       for i in range(3)] for q in range(2)])
    np.testing.assert_allclose(Sg, brute, rtol=1e-12)
    np.testing.assert_allclose(Sm, brute, rtol=1e-12)


def test_identity_projection_scores_equal_exact_similarity(orc):
    rng = np.random.default_rng(8)
    T, d = 4, 6
    Aq, Bq = _rand(rng, 2, T, d), _rand(rng, 2, T, d)
    At, Bt = _rand(rng, 5, T, d), _rand(rng, 5, T, d)
    fq = orc.project(Aq, Bq, d, d, seed=0, layer=0, kind=1)
    ft = orc.project(At, Bt, d, d, seed=0, layer=0, kind=1)
    np.testing.assert_allclose(orc.score(fq, ft), orc.similarity(Aq, Bq, At, Bt), rtol=1e-12)


def test_gram_on_projected_factors_equals_projected_scores(orc):
    # Projected factors keep the Eq. 1 form (App. A.2), so Eq. 4 applies to them.
    rng = np.random.default_rng(9)
    T, d_in, d_out, k_in, k_out = 5, 16, 12, 4, 8
    Aq, Bq = _rand(rng, 2, T, d_in), _rand(rng, 2, T, d_out)
    At, Bt = _rand(rng, 3, T, d_in), _rand(rng, 3, T, d_out)
    P_in = orc.proj_matrix(3, 7, 0, d_in, k_in)
    P_out = orc.proj_matrix(3, 7, 1, d_out, k_out)
    fq = orc.project(Aq, Bq, k_in, k_out, seed=3, layer=7)
    ft = orc.project(At, Bt, k_in, k_out, seed=3, layer=7)
    Sg = orc.similarity(Aq @ P_in, Bq @ P_out, At @ P_in, Bt @ P_out, route="gram")
    np.testing.assert_allclose(orc.score(fq, ft), Sg, rtol=1e-12)


def test_squared_norms_two_routes_and_brute_force(orc):
    # App. A.4 routes norms like Gram matrices: ||DW||^2 by Eq. 1 and by Eq. 4 agree
    rng = np.random.default_rng(10)
    N, T, di, do = 4, 6, 9, 7
    A, B = _rand(rng, N, T, di), _rand(rng, N, T, do)
    g = orc.sq_norms(A, B, "gram")
    m = orc.sq_norms(A, B, "materialized")
    brute = np.array([float((orc.materialize(A[n], B[n]) ** 2).sum()) for n in range(N)])
    np.testing.assert_allclose(g, brute, rtol=1e-12)
    np.testing.assert_allclose(m, brute, rtol=1e-12)
    # a rank-one gradient g a^T (T = 1) has norm ||g||^2 ||a||^2
    one = orc.sq_norms(A[:, :1], B[:, :1])
    np.testing.assert_allclose(one, (A[:, 0] ** 2).sum(1) * (B[:, 0] ** 2).sum(1), rtol=1e-13)


def test_cosine_properties(orc):
    rng = np.random.default_rng(11)
    X = rng.standard_normal((5, 12))
    S = orc.score(X, X)
    n = (X ** 2).sum(1)
    C = orc.cosine(S, n, n)
    np.testing.assert_allclose(np.diag(C), 1.0, rtol=1e-14)
    assert np.abs(C).max() <= 1 + 1e-12
    # invariant to scaling either side
    C2 = orc.cosine(orc.score(3 * X, X), 9 * n, n)
    np.testing.assert_allclose(C2, C, rtol=1e-13)
