"""Pins for the oracle's route cost model (Sec. 3.2 routing, App. A.4 Table 2)."""
import numpy as np
import pytest


def test_exact_similarity_counts_closed_form(orc):
    # Table 2, 2 flops per multiply-add:
    # factorised 2 B1 B2 T^2 (N_i + N_o); materialised 2 (B1+B2) T N_i N_o + 2 B1 B2 N_i N_o
    best, c = orc.route_costs(orc.OP_SIM_EXACT, 3, 5, 7, 11, 13)
    assert c[0] == -1
    assert c[1] == 2 * 8 * 7 * 11 * 13 + 2 * 15 * 11 * 13
    assert c[2] == 2 * 15 * 49 * (11 + 13)
    assert best == (2 if c[2] <= c[1] else 1)


def test_project_counts_closed_form(orc):
    N, T, di, do, ki, ko = 4, 10, 32, 48, 8, 16
    best, c = orc.route_costs(orc.OP_PROJECT, N, 0, T, di, do, ki, ko)
    assert c[0] == N * (2 * T * (di * ki + do * ko) + 2 * T * ki * ko)
    assert c[1] == N * (2 * T * di * do + 2 * do * di * ki + 2 * do * ki * ko)
    assert c[2] == -1
    assert best == 0


def test_crossover_of_square_layer_matches_paper_regimes(orc):
    # App. A.4 regimes and App. B.4: for full-dimensional comparison of one
    # query with a batch of 8, short sequences favour the factorised route and
    # long ones materialisation. For a square 1024-wide layer the two counts
    # cross near T = 576 (between the paper's T = 512 and T = 2048 points).
    for T, want in [(32, 2), (128, 2), (512, 2), (2048, 1)]:
        best, _ = orc.route_costs(orc.OP_SIM_EXACT, 1, 8, T, 1024, 1024)
        assert best == want, T
    lo = max(T for T in range(1, 4096) if orc.route_costs(orc.OP_SIM_EXACT, 1, 8, T, 1024, 1024)[0] == 2)
    assert 570 <= lo <= 580


def test_projection_shrinks_the_factorised_regime(orc):
    # Under factor projection N_i, N_o become k_a, k_g (App. A.4): for a wide layer
    # at T = 512 the projected Gram route loses to materialising k x k features.
    best, c = orc.route_costs(orc.OP_SIM_PROJECTED, 64, 4096, 512, 2048, 2048, 32, 32)
    assert best == 0
    assert c[2] > c[0] and c[1] > c[0]


@pytest.mark.parametrize("T", [1, 4])
def test_tiny_T_prefers_gram_for_projected_similarity(orc, T):
    best, _ = orc.route_costs(orc.OP_SIM_PROJECTED, 8, 8, T, 256, 256, 64, 64)
    assert best == 2


def test_norm_costs_are_table2_with_one_example_per_side(orc):
    n, T, di, do, k = 5, 16, 64, 32, 8
    _, c = orc.route_costs(orc.OP_NORM_EXACT, n, 0, T, di, do)
    assert c[0] == -1
    assert c[1] == n * (2 * T * di * do + 2 * di * do)
    assert c[2] == n * 2 * T * T * (di + do)
    _, cp = orc.route_costs(orc.OP_NORM_PROJECTED, n, 0, T, di, do, k, k)
    assert cp[2] == n * (2 * T * (di * k + do * k) + 2 * T * T * (2 * k))
    # long sequences favour materialising for exact norms, short ones the Gram route
    assert orc.route_costs(orc.OP_NORM_EXACT, 1, 0, 4, 1024, 1024)[0] == 2
    assert orc.route_costs(orc.OP_NORM_EXACT, 1, 0, 4096, 1024, 1024)[0] == 1


# ---------------------------------------------------------------------------
# Counted loop nests. Each route of each op is carried out below on tiny
# shapes with explicit loops that count every multiply-add of the contractions
# Table 2 prices (2 flops each); the results are checked against the oracle's
# own routines, so the counted loops are the real computation. A dropped or
# doubled term in oracle_route_costs fails the count.

B1, B2, TT, DI, DO, KI, KO = 2, 3, 3, 4, 5, 2, 3


class _Count:
    def __init__(self):
        self.macs = 0

    def mm(self, X, Y):
        """X (m, k) @ Y (k, n) with explicit loops."""
        m, k = X.shape
        n = Y.shape[1]
        out = np.zeros((m, n))
        for i in range(m):
            for j in range(n):
                s = 0.0
                for l in range(k):
                    s += X[i, l] * Y[l, j]
                    self.macs += 1
                out[i, j] = s
        return out

    def dot(self, x, y):
        s = 0.0
        for a, b in zip(x.ravel(), y.ravel()):
            s += a * b
            self.macs += 1
        return s


def _factors(n, seed):
    rng = np.random.default_rng(seed)
    return rng.standard_normal((n, TT, DI)), rng.standard_normal((n, TT, DO))


def _maps(orc):
    return orc.proj_matrix(0, 0, 0, DI, KI), orc.proj_matrix(0, 0, 1, DO, KO)


def _proj_factored(c, A, B, Pin, Pout):
    """Route (a): a~ = A P_in, g~ = B P_out, Phi = g~^T a~ (k_out x k_in)."""
    At, Bt = c.mm(A, Pin), c.mm(B, Pout)
    return At, Bt, c.mm(Bt.T, At)


def _proj_materialized(c, A, B, Pin, Pout):
    """Route (b): DW = B^T A, then P_out^T (DW P_in)."""
    G = c.mm(B.T, A)
    return c.mm(Pout.T, c.mm(G, Pin))


def test_projection_and_projected_similarity_costs_count_loop_nests(orc):
    Aq, Bq = _factors(B1, 1)
    At, Bt = _factors(B2, 2)
    Pin, Pout = _maps(orc)
    ref = orc.project(np.concatenate([Aq, At]), np.concatenate([Bq, Bt]), KI, KO, 0, 0)
    # op 0 over the B1 query examples, both routes
    ca, cb = _Count(), _Count()
    for e in range(B1):
        _, _, phi_a = _proj_factored(ca, Aq[e], Bq[e], Pin, Pout)
        phi_b = _proj_materialized(cb, Aq[e], Bq[e], Pin, Pout)
        np.testing.assert_allclose(phi_a, ref[e], rtol=1e-12, atol=1e-12)
        np.testing.assert_allclose(phi_b, ref[e], rtol=1e-12, atol=1e-12)
    _, c0 = orc.route_costs(orc.OP_PROJECT, B1, 0, TT, DI, DO, KI, KO)
    assert c0[0] == 2 * ca.macs and c0[1] == 2 * cb.macs
    # op 1: B1 x B2 similarities of projected gradients by all three routes
    ca, cb, cg = _Count(), _Count(), _Count()
    fa, fb, fac = [], [], []
    for A, B in [(Aq[e], Bq[e]) for e in range(B1)] + [(At[e], Bt[e]) for e in range(B2)]:
        fa.append(_proj_factored(ca, A, B, Pin, Pout)[2])
        fb.append(_proj_materialized(cb, A, B, Pin, Pout))
        at, bt = cg.mm(A, Pin), cg.mm(B, Pout)  # route (c) keeps the projected factors
        fac.append((at, bt))
    Sa = np.array([[ca.dot(fa[q], fa[B1 + i]) for i in range(B2)] for q in range(B1)])
    Sb = np.array([[cb.dot(fb[q], fb[B1 + i]) for i in range(B2)] for q in range(B1)])
    prod_sum = 0
    Sg = np.zeros((B1, B2))
    for q in range(B1):
        for i in range(B2):
            X = cg.mm(fac[q][0], fac[B1 + i][0].T)  # T x T token Gram of a~
            Y = cg.mm(fac[q][1], fac[B1 + i][1].T)  # T x T token Gram of g~
            Sg[q, i] = float((X * Y).sum())  # Eq. 4's elementwise product-sum
            prod_sum += TT * TT
    Sref = ref[:B1].reshape(B1, -1) @ ref[B1:].reshape(B2, -1).T
    for S in (Sa, Sb, Sg):
        np.testing.assert_allclose(S, Sref, rtol=1e-11, atol=1e-11)
    _, c1 = orc.route_costs(orc.OP_SIM_PROJECTED, B1, B2, TT, DI, DO, KI, KO)
    assert c1[0] == 2 * ca.macs
    assert c1[1] == 2 * cb.macs
    # Table 2 prices the two token-Gram contractions; the T^2 product-sum per pair is not in its count
    assert c1[2] == 2 * cg.macs
    assert prod_sum == B1 * B2 * TT * TT


def test_exact_similarity_and_norm_costs_count_loop_nests(orc):
    Aq, Bq = _factors(B1, 3)
    At, Bt = _factors(B2, 4)
    # op 2: materialise every DW, then Frobenius dots; or the Gram identity per pair
    cb, cg = _Count(), _Count()
    G = [cb.mm(B.T, A) for A, B in [(Aq[e], Bq[e]) for e in range(B1)] + [(At[e], Bt[e]) for e in range(B2)]]
    Sb = np.array([[cb.dot(G[q], G[B1 + i]) for i in range(B2)] for q in range(B1)])
    Sg = np.array([[float((cg.mm(Aq[q], At[i].T) * cg.mm(Bq[q], Bt[i].T)).sum()) for i in range(B2)]
                   for q in range(B1)])
    ref = orc.similarity(Aq, Bq, At, Bt)
    np.testing.assert_allclose(Sb, ref, rtol=1e-11)
    np.testing.assert_allclose(Sg, ref, rtol=1e-11)
    _, c2 = orc.route_costs(orc.OP_SIM_EXACT, B1, B2, TT, DI, DO)
    assert c2[1] == 2 * cb.macs and c2[2] == 2 * cg.macs
    # op 4: exact squared norms of the B1 examples, materialised or by the Gram identity
    cb, cg = _Count(), _Count()
    nb = [cb.dot(*(2 * [cb.mm(Bq[e].T, Aq[e])])) for e in range(B1)]
    ng = [float((cg.mm(Aq[e], Aq[e].T) * cg.mm(Bq[e], Bq[e].T)).sum()) for e in range(B1)]
    np.testing.assert_allclose(nb, orc.sq_norms(Aq, Bq), rtol=1e-12)
    np.testing.assert_allclose(ng, orc.sq_norms(Aq, Bq), rtol=1e-12)
    _, c4 = orc.route_costs(orc.OP_NORM_EXACT, B1, 0, TT, DI, DO)
    assert c4[1] == 2 * cb.macs and c4[2] == 2 * cg.macs
    # op 3: squared norms of the projected gradients by the three routes
    Pin, Pout = _maps(orc)
    ca, cb, cg = _Count(), _Count(), _Count()
    na, nb, ng = [], [], []
    for e in range(B1):
        phi = _proj_factored(ca, Aq[e], Bq[e], Pin, Pout)[2]
        na.append(ca.dot(phi, phi))
        phi = _proj_materialized(cb, Aq[e], Bq[e], Pin, Pout)
        nb.append(cb.dot(phi, phi))
        at, bt = cg.mm(Aq[e], Pin), cg.mm(Bq[e], Pout)
        ng.append(float((cg.mm(at, at.T) * cg.mm(bt, bt.T)).sum()))
    ref = (orc.project(Aq, Bq, KI, KO, 0, 0).reshape(B1, -1) ** 2).sum(1)
    for n in (na, nb, ng):
        np.testing.assert_allclose(n, ref, rtol=1e-12)
    _, c3 = orc.route_costs(orc.OP_NORM_PROJECTED, B1, 0, TT, DI, DO, KI, KO)
    assert c3[0] == 2 * ca.macs and c3[1] == 2 * cb.macs and c3[2] == 2 * cg.macs


def test_exact_ties_prefer_gram_then_the_factored_projection(orc):
    # The tie rule (a reading: App. A.4 prefers the factorised form for its memory): on equal
    # counts the Gram route wins, then the factored projection, then materialisation.
    # Projected similarity ties exactly at B1 = 1, B2 = 2, T = 2, k_a = k_g = 2: beyond the
    # shared projection of the factors the factored route adds (B1+B2) 2 T k_a k_g + B1 B2 2 k_a k_g
    # = 48 + 16 and the Gram route B1 B2 2 T^2 (k_a + k_g) = 64.
    best, c = orc.route_costs(orc.OP_SIM_PROJECTED, 1, 2, 2, 64, 64, 2, 2)
    assert c[0] == c[2] < c[1] and best == 2
    # Projection ties at T = d_in = d_out = k = 1: factored 2T(d k + d k) + 2T k^2 = 6,
    # materialised 2T d^2 + 2 d^2 k + 2 d k^2 = 6.
    best, c = orc.route_costs(orc.OP_PROJECT, 1, 0, 1, 1, 1, 1, 1)
    assert c[0] == c[1] == 6 and best == 0
