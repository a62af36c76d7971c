"""C-ABI checks that need no GPU: the library builds and loads, exports every
declared symbol, validates arguments on the host, and its host-only route
cost model agrees with the oracle's (App. A.4, Table 2)."""
import ctypes
import os
import re

import numpy as np
import pytest

import paper_2609_38767_gb300 as tda
from paper_2609_38767_gb300 import build as tbuild

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def libs():
    return tbuild.build()


def _declared(header):
    text = open(os.path.join(ROOT, "include", header)).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(tda_\w+)\s*\(", text)))


@pytest.mark.parametrize("header,lib", [("tda.h", "libtda.so"), ("tda_synth.h", "libtda_synth.so")])
def test_every_declared_symbol_is_exported(libs, header, lib):
    so = ctypes.CDLL(libs[lib])
    names = _declared(header)
    assert names, header
    missing = [n for n in names if not hasattr(so, n)]
    assert not missing, missing


def test_layer_desc_layout_matches_header():
    assert ctypes.sizeof(tda.LayerDesc) == 48
    assert tda.LayerDesc.seed.offset == 32 and tda.LayerDesc.kind.offset == 44


def test_version_and_state_bytes(libs):
    assert tda.tda_version() >= 100
    def rup(x):
        return (x + 255) // 256 * 256
    assert tda.tda_precondition_state_bytes(256, tda.TDA_F64) == rup(64 + (256 * 256 + 8 * 1024) * 8)
    assert tda.tda_precondition_state_bytes(10, tda.TDA_F32) == rup(64 + (100 + 1024) * 4)
    assert tda.tda_precondition_state_bytes(0, tda.TDA_F32) == 0


def _err(fn, *a, **k):
    with pytest.raises(tda.TdaError) as e:
        fn(*a, **k)
    return e.value.status


def test_host_validation_rejects_bad_arguments(libs):
    L = tda.LayerDesc(64, 64, 8, 16, 16)
    s = 0  # never reached: validation fails first
    assert _err(tda.tda_project, L, tda.TDA_BF16, None, None, 4, None, 256, stream=s) == tda.TDA_ERR_INVALID_ARG
    assert _err(tda.tda_project, L, tda.TDA_BF16, 16, 16, 4, 16, 100, stream=s) == tda.TDA_ERR_INVALID_ARG
    assert _err(tda.tda_project, L, tda.TDA_BF16, 8, 16, 4, 16, 256, stream=s) == tda.TDA_ERR_INVALID_ARG
    assert _err(tda.tda_project, L, 7, 16, 16, 4, 16, 256, stream=s) == tda.TDA_ERR_INVALID_ARG
    bad = tda.LayerDesc(60, 64, 8, 16, 16)  # d_in not a multiple of 8 for bf16
    assert _err(tda.tda_project, bad, tda.TDA_BF16, 16, 16, 4, 16, 256, stream=s) == tda.TDA_ERR_INVALID_ARG
    ident = tda.LayerDesc(64, 64, 8, 16, 16, kind=tda.TDA_PROJ_IDENTITY)
    assert _err(tda.tda_project, ident, tda.TDA_F32, 16, 16, 4, 16, 256, stream=s) == tda.TDA_ERR_INVALID_ARG
    assert _err(tda.tda_project, L, tda.TDA_BF16, 16, 16, 4, 16, 256, route=tda.TDA_ROUTE_MATERIALIZE,
                ws=None, ws_bytes=0, stream=s) == tda.TDA_ERR_WORKSPACE
    assert _err(tda.tda_project, L, tda.TDA_BF16, 16, 16, 4, 16, 256, route=tda.TDA_ROUTE_GRAM,
                stream=s) == tda.TDA_ERR_UNSUPPORTED
    assert _err(tda.tda_topk, 16, 2, 10, 10, 11, 16, stream=s) == tda.TDA_ERR_INVALID_ARG
    assert _err(tda.tda_topk, 16, 2, 10, 10, 0, 16, stream=s) == tda.TDA_ERR_INVALID_ARG
    assert _err(tda.tda_score, 16, tda.TDA_BF16, 2, 8, 16, 3, 8, 8, 16, 3, stream=s) == tda.TDA_ERR_INVALID_ARG
    assert _err(tda.tda_score, 16, tda.TDA_F32, 2, 4, 16, 3, 8, 8, 16, 3, stream=s) == tda.TDA_ERR_INVALID_ARG
    assert _err(tda.tda_precondition, 9, 1, 8, tda.TDA_F64, 16, stream=s) == tda.TDA_ERR_INVALID_ARG
    assert _err(tda.tda_precondition, tda.TDA_PC_RESET, 0, 8, tda.TDA_F64, 16, stream=s) == tda.TDA_ERR_INVALID_ARG
    assert _err(tda.tda_precondition, tda.TDA_PC_FIT_ACCUM, 3, 8, tda.TDA_F32, 16, phi=16, n=4, ld_phi=16,
                stream=s) == tda.TDA_ERR_INVALID_ARG  # ld_phi < 3*8
    assert _err(tda.tda_precondition, tda.TDA_PC_APPLY, 1, 50000, tda.TDA_F32, 16, q=16, n_q=1, ld_q=50000,
                qhat=16, ld_qhat=50000, stream=s) == tda.TDA_ERR_UNSUPPORTED
    assert _err(tda.tda_precondition, tda.TDA_PC_FACTOR, 1, 8, tda.TDA_F64, 16, n_total=0, lambda_abs=1.0,
                stream=s) == tda.TDA_ERR_INVALID_ARG
    assert _err(tda.tda_precondition, tda.TDA_PC_FACTOR, 1, 8, tda.TDA_F64, 16, n_total=4, stream=s) \
        == tda.TDA_ERR_INVALID_ARG
    assert _err(tda.tda_proj_entries, 0, 0, 2, 0, 4, 4, 16, stream=s) == tda.TDA_ERR_INVALID_ARG
    assert _err(tda.tda_route_set_model, 1) == tda.TDA_ERR_INVALID_ARG
    assert _err(tda.tda_route_calibrate, None, 0, stream=s) == tda.TDA_ERR_WORKSPACE
    assert "ws" in tda.tda_last_error()


SHAPES = [
    # (n1, n2, T, d_in, d_out, k_in, k_out)
    (1, 8, 32, 1024, 1024, 64, 64), (1, 8, 2048, 1024, 1024, 64, 64), (64, 4096, 512, 2048, 8192, 32, 32),
    (128, 2 ** 24 // 8, 8, 8192, 8192, 64, 64), (128, 2 ** 24 // 8192, 8192, 8192, 8192, 64, 64),
    (8, 64, 32, 256, 256, 16, 16), (3, 5, 1, 24, 40, 8, 8), (512, 16384, 2048, 12288, 49152, 128, 128),
    # exact ties of the Table 2 counts (projected similarity: factored = Gram; projection: factored =
    # materialised): the library breaks them as the oracle does
    (1, 2, 2, 64, 64, 2, 2), (1, 0, 1, 1, 1, 1, 1),
]


@pytest.mark.parametrize("shape", SHAPES)
@pytest.mark.parametrize("op", [tda.TDA_OP_PROJECT, tda.TDA_OP_SIMILARITY_PROJECTED, tda.TDA_OP_SIMILARITY_EXACT,
                                tda.TDA_OP_NORM_PROJECTED, tda.TDA_OP_NORM_EXACT])
def test_route_flop_model_matches_oracle(libs, orc, shape, op):
    n1, n2, T, di, do, ki, ko = shape
    L = tda.LayerDesc(di, do, T, ki, ko)
    chosen, cost = tda.tda_route(L, op, n1, n2, tda.TDA_BF16)
    best, ocost = orc.route_costs(op, n1, n2, T, di, do, ki, ko)
    assert chosen == best
    np.testing.assert_allclose(cost, ocost, rtol=1e-12)


def test_workspace_sizes(libs):
    L = tda.LayerDesc(256, 128, 32, 16, 16)
    assert tda.tda_workspace_size(tda.TDA_OP_PROJECT, L, tda.TDA_F32, 10, 0, tda.TDA_ROUTE_FACTORED) == 0
    assert tda.tda_workspace_size(tda.TDA_OP_PROJECT, L, tda.TDA_F32, 10, 0,
                                  tda.TDA_ROUTE_MATERIALIZE) == 4 * (128 * 256 + 128 * 16)
    # the 3 query DW, one train DW and the split-K partials of 3 dots over at most 256 slices
    assert tda.tda_workspace_size(tda.TDA_OP_SIMILARITY_EXACT, L, tda.TDA_F32, 3, 9,
                                  tda.TDA_ROUTE_MATERIALIZE) == 4 * (4 * 128 * 256 + 256 * 3)
    assert tda.tda_workspace_size(tda.TDA_OP_SIMILARITY_EXACT, L, tda.TDA_F32, 3, 9, tda.TDA_ROUTE_GRAM) == 0
    D = 16 * 16
    assert tda.tda_workspace_size(tda.TDA_OP_SIMILARITY_PROJECTED, L, tda.TDA_F32, 3, 9,
                                  tda.TDA_ROUTE_FACTORED) == 4 * D * 4
    assert tda.tda_workspace_size(tda.TDA_OP_SIMILARITY_PROJECTED, L, tda.TDA_F32, 3, 9,
                                  tda.TDA_ROUTE_MATERIALIZE) == 4 * D * 4 + 4 * (128 * 256 + 128 * 16)
    assert tda.tda_workspace_size(tda.TDA_OP_SIMILARITY_PROJECTED, L, tda.TDA_F32, 3, 9,
                                  tda.TDA_ROUTE_GRAM) == 4 * 32 * (16 + 16) * 4
    # norms: one example at a time per chunk
    assert tda.tda_workspace_size(tda.TDA_OP_NORM_PROJECTED, L, tda.TDA_F32, 3, 0, tda.TDA_ROUTE_FACTORED) == 4 * D
    assert tda.tda_workspace_size(tda.TDA_OP_NORM_PROJECTED, L, tda.TDA_F32, 3, 0,
                                  tda.TDA_ROUTE_MATERIALIZE) == 4 * D + 4 * (128 * 256 + 128 * 16)
    assert tda.tda_workspace_size(tda.TDA_OP_NORM_PROJECTED, L, tda.TDA_F32, 3, 0,
                                  tda.TDA_ROUTE_GRAM) == 4 * 32 * (16 + 16)
    assert tda.tda_workspace_size(tda.TDA_OP_NORM_EXACT, L, tda.TDA_F32, 3, 0,
                                  tda.TDA_ROUTE_MATERIALIZE) == 4 * 128 * 256
    assert tda.tda_workspace_size(tda.TDA_OP_NORM_EXACT, L, tda.TDA_F32, 3, 0, tda.TDA_ROUTE_GRAM) == 0


def test_norm_entry_validation(libs):
    L = tda.LayerDesc(64, 64, 8, 16, 16)
    s = 0
    assert _err(tda.tda_norms, tda.TDA_OP_PROJECT, L, tda.TDA_F32, 16, 16, 4, 16, stream=s) \
        == tda.TDA_ERR_INVALID_ARG
    assert _err(tda.tda_norms, tda.TDA_OP_NORM_EXACT, L, tda.TDA_F32, 16, 16, 4, 16,
                route=tda.TDA_ROUTE_FACTORED, stream=s) == tda.TDA_ERR_UNSUPPORTED
    assert _err(tda.tda_norms, tda.TDA_OP_NORM_PROJECTED, L, tda.TDA_F32, 16, 16, 4, 16,
                route=tda.TDA_ROUTE_FACTORED, stream=s) == tda.TDA_ERR_WORKSPACE
    assert _err(tda.tda_norms, tda.TDA_OP_NORM_PROJECTED, L, tda.TDA_F32, 16, 16, 4, None, stream=s) \
        == tda.TDA_ERR_INVALID_ARG
    assert _err(tda.tda_cosine, 16, 2, 8, 4, 16, 16, stream=s) == tda.TDA_ERR_INVALID_ARG


def test_kfac_state_and_validation(libs):
    # state: 8-double header + Sa, Sg, Ua, wa, Ug, wg, EK-FAC sums (fp64), 256-byte multiple
    for ka, kg in [(16, 16), (32, 64), (128, 128), (1, 3)]:
        n = 8 + 2 * ka * ka + ka + 2 * kg * kg + kg + ka * kg
        assert tda.tda_kfac_state_bytes(ka, kg) == (n * 8 + 255) // 256 * 256
    assert tda.tda_kfac_state_bytes(0, 16) == 0 and tda.tda_kfac_state_bytes(16, 129) == 0
    L = tda.LayerDesc(64, 64, 8, 16, 16)
    s = 0
    assert _err(tda.tda_kfac_reset, 16, 200, 256, stream=s) == tda.TDA_ERR_INVALID_ARG
    assert _err(tda.tda_kfac_reset, 16, 16, 8, stream=s) == tda.TDA_ERR_INVALID_ARG  # misaligned state
    assert _err(tda.tda_kfac_apply, 2, 16, 16, 256, 0.0, 0.1, 256, 1, 256, 256, 256, stream=s) \
        == tda.TDA_ERR_INVALID_ARG
    assert _err(tda.tda_kfac_apply, tda.TDA_KFAC, 16, 16, 256, 0.0, 0.1, 256, 1, 100, 256, 256, stream=s) \
        == tda.TDA_ERR_INVALID_ARG  # ld_q < 256
    assert _err(tda.tda_kfac_accumulate_factors, L, tda.TDA_BF16, 16, 16, 4, 256, 256, 100, stream=s) \
        == tda.TDA_ERR_WORKSPACE
    assert _err(tda.tda_kfac_accumulate_eigenvalues, 16, 16, 256, 16, 4, 256, 256, 100, stream=s) \
        == tda.TDA_ERR_WORKSPACE
    assert _err(tda.tda_project_kfac, L, tda.TDA_F32, 16, 16, 4, 16, 256, 256, 256, 1 << 24, stream=s) \
        == tda.TDA_ERR_UNSUPPORTED


def test_sm_budget_is_host_state(libs):
    # the projection's SM cap is plain host state: set, read back, reset; negative rejected
    assert tda.tda_get_sm_budget() == 0
    tda.tda_set_sm_budget(100)
    assert tda.tda_get_sm_budget() == 100
    assert _err(tda.tda_set_sm_budget, -1) == tda.TDA_ERR_INVALID_ARG
    assert tda.tda_get_sm_budget() == 100
    tda.tda_set_sm_budget(0)
    assert tda.tda_get_sm_budget() == 0


@pytest.mark.parametrize("k", [16, 32, 64, 128])
def test_factored_projection_workspace_layout(libs, k):
    # bf16 factored projection: the optional workspace is [k = 128 sign tables, rounded up to
    # 256 bytes][two k x k fp32 partial blocks and one counter per SM]; any other k or dtype
    # needs none
    di, do = 1000, 2056
    L = tda.LayerDesc(di, do, 300, k, k)
    b = tda.tda_workspace_size(tda.TDA_OP_PROJECT, L, tda.TDA_BF16, 7, 0, tda.TDA_ROUTE_FACTORED)
    signs = (2 * k * (di + do) + 255) // 256 * 256 if k == 128 else 0
    per_sm = 2 * k * k * 4 + 4
    assert b > signs and (b - signs) % per_sm == 0
    L2 = tda.LayerDesc(di, do, 300, k, k // 2 if k > 16 else 32)
    assert tda.tda_workspace_size(tda.TDA_OP_PROJECT, L2, tda.TDA_BF16, 7, 0, tda.TDA_ROUTE_FACTORED) == 0
    assert tda.tda_workspace_size(tda.TDA_OP_PROJECT, L, tda.TDA_F32, 7, 0, tda.TDA_ROUTE_FACTORED) == 0


def test_route_model_matches_oracle_on_random_shapes(libs, orc):
    # 600 seeded random shapes over every op (the flop model does not depend on the dtype):
    # the library's host-side cost model and choice equal the oracle's Table 2 counts
    rng = np.random.default_rng(7)
    for _ in range(600):
        op = int(rng.integers(0, 5))
        n1, n2 = int(rng.integers(0, 5000)), int(rng.integers(0, 5000))
        T = int(2 ** rng.integers(0, 14)) if rng.random() < 0.5 else int(rng.integers(1, 9000))
        di, do = int(rng.integers(1, 20000)), int(rng.integers(1, 20000))
        ki, ko = int(rng.integers(1, 257)), int(rng.integers(1, 257))
        L = tda.LayerDesc(di, do, T, ki, ko)
        chosen, cost = tda.tda_route(L, op, n1, n2, tda.TDA_BF16)
        best, ocost = orc.route_costs(op, n1, n2, T, di, do, ki, ko)
        assert chosen == best, (op, n1, n2, T, di, do, ki, ko, cost, ocost)
        np.testing.assert_allclose(cost, ocost, rtol=1e-12)
