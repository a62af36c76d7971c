"""Pins for the oracle's route cost model (Sec. 3.2 routing, App. A.4 Table 2)."""
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
