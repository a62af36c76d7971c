"""Pins for the oracle's token-level scores (token-level attribution appendix)
and random-mask reduction (masked coordinates of Eq. 1)."""
import numpy as np
import pytest


def test_token_scores_sum_to_the_sequence_score(orc):
    # sum_t s_t = <Phi_i, R_j> (the decomposition's defining identity)
    rng = np.random.default_rng(0)
    N, T, di, do, k, nq = 3, 7, 24, 16, 8, 2
    A, B = rng.standard_normal((N, T, di)), rng.standard_normal((N, T, do))
    R = rng.standard_normal((nq, k, k))
    s = orc.token_scores(A, B, R, k, k, seed=4, layer=2)
    phi = orc.project(A, B, k, k, seed=4, layer=2)
    np.testing.assert_allclose(s.sum(2), orc.score(R, phi), rtol=1e-12)


def test_token_scores_identity_map_brute_force(orc):
    # identity projection: s_t = g_t^T R a_t with R a full d_out x d_in matrix
    rng = np.random.default_rng(1)
    N, T, d = 2, 5, 6
    A, B = rng.standard_normal((N, T, d)), rng.standard_normal((N, T, d))
    R = rng.standard_normal((3, d, d))
    s = orc.token_scores(A, B, R, d, d, seed=0, layer=0, kind=1)
    brute = np.einsum("itr,jrc,itc->jit", B, R, A)
    np.testing.assert_allclose(s, brute, rtol=1e-12, atol=1e-12)
    # a masked (zero) token contributes nothing
    A[0, 2] = 0.0
    assert orc.token_scores(A, B, R, d, d, seed=0, layer=0, kind=1)[:, 0, 2].tolist() == [0.0] * 3


def test_mask_gather_is_dw_at_the_coordinates(orc):
    rng = np.random.default_rng(2)
    N, T, di, do = 3, 9, 20, 12
    A, B = rng.standard_normal((N, T, di)), rng.standard_normal((N, T, do))
    flat = rng.permutation(di * do)[:30]
    rows, cols = flat // di, flat % di
    got = orc.mask_gather(A, B, rows, cols)
    for n in range(N):
        G = orc.materialize(A[n], B[n])
        np.testing.assert_allclose(got[n], G[rows, cols], rtol=1e-13)


def test_disjoint_masks_average_equals_concatenated_inner_product(orc):
    # scores of ten disjoint masks, averaged, equal one score over the union / 10
    rng = np.random.default_rng(3)
    N, T, d, k, n_masks = 4, 6, 16, 5, 10
    A, B = rng.standard_normal((N, T, d)), rng.standard_normal((N, T, d))
    Aq, Bq = rng.standard_normal((2, T, d)), rng.standard_normal((2, T, d))
    flat = rng.permutation(d * d)[: n_masks * k].reshape(n_masks, k)
    per_mask = []
    for m in range(n_masks):
        r, c = flat[m] // d, flat[m] % d
        per_mask.append(orc.score(orc.mask_gather(Aq, Bq, r, c), orc.mask_gather(A, B, r, c)))
    r, c = flat.reshape(-1) // d, flat.reshape(-1) % d
    union = orc.score(orc.mask_gather(Aq, Bq, r, c), orc.mask_gather(A, B, r, c))
    np.testing.assert_allclose(np.mean(per_mask, 0), union / n_masks, rtol=1e-12)
