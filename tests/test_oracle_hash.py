"""Pins for the oracle's projection-sign hash (App. A.2 random maps, seeds per layer and side)."""
import os

import numpy as np
import pytest

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _golden_words(name):
    with open(os.path.join(GOLDEN, name)) as f:
        return [int(line, 16) for line in f if line.strip() and not line.startswith("#")]


def test_splitmix64_reference_vector(orc):
    # the mixer must reproduce the generator's published outputs
    assert orc.splitmix64_sequence(0, 3) == _golden_words("splitmix64_seed0.txt")


def test_mix64_is_bijective_on_sample(orc):
    xs = [orc.mix64(i) for i in range(4096)]
    assert len(set(xs)) == 4096
    assert orc.mix64(0) == 0  # xor-shift-multiply fixes zero; the counter offset avoids it


def test_sign_entries_are_pm1_and_shape_independent(orc):
    a = orc.proj_entries(7, 3, 0, 100, 10)
    b = orc.proj_entries(7, 3, 0, 200, 20)
    assert set(np.unique(a)) <= {-1, 1}
    assert np.array_equal(a, b[:100, :10])
    assert orc.proj_sign(7, 3, 0, 57, 4) == a[57, 4]


def test_sign_balance_and_independence(orc):
    rows, cols = 4096, 64
    S = orc.proj_entries(0, 0, 0, rows, cols).astype(np.float64)
    n = rows * cols
    # fraction of +1 within 4 sigma of 1/2
    frac = (S > 0).mean()
    assert abs(frac - 0.5) < 4 * 0.5 / np.sqrt(n)
    # pairwise column correlations of independent signs: sd 1/sqrt(rows)
    C = (S.T @ S) / rows
    off = C[~np.eye(cols, dtype=bool)]
    assert np.abs(off).max() < 5.5 / np.sqrt(rows)
    assert abs(off.mean()) < 4 / np.sqrt(rows * off.size)
    # row correlations within one 64-row hash block are independent too
    R = (S[:64] @ S[:64].T) / cols
    offr = R[~np.eye(64, dtype=bool)]
    assert np.abs(offr).max() < 6 / np.sqrt(cols)


def test_layers_and_sides_use_distinct_streams(orc):
    base = orc.proj_entries(0, 0, 0, 512, 32)
    for other in (orc.proj_entries(0, 0, 1, 512, 32), orc.proj_entries(0, 1, 0, 512, 32),
                  orc.proj_entries(1, 0, 0, 512, 32)):
        agree = (base == other).mean()
        assert abs(agree - 0.5) < 4 * 0.5 / np.sqrt(base.size)


def test_identity_kind(orc):
    E = orc.proj_entries(5, 2, 1, 24, 24, kind=1)
    assert np.array_equal(E, np.eye(24, dtype=np.int8))
    P = orc.proj_matrix(5, 2, 1, 24, 24, kind=1)
    assert np.array_equal(P, np.eye(24))


@pytest.mark.parametrize("k", [1, 16, 32, 100])
def test_rademacher_scale_is_inverse_sqrt_output_dim(orc, k):
    P = orc.proj_matrix(11, 4, 0, 300, k)
    assert np.allclose(np.abs(P), 1.0 / np.sqrt(k), rtol=0, atol=0)
    E = orc.proj_entries(11, 4, 0, 300, k)
    assert np.array_equal(np.sign(P).astype(np.int8), E)
