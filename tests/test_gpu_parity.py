"""GPU parity: every entry point of libtda.so, called through the C ABI, against
the fp64 oracle on the same seeded inputs. Tolerances: projected features and
score matrices within a relative Frobenius error of 1e-5 for fp32 factors and
2e-2 for bf16 factors (fp32 accumulation); sign entries, indices and top-k
bit-exact."""
import os

import numpy as np
import pytest
import torch

import paper_2609_38767_gb300 as tda
from paper_2609_38767_gb300 import build as tbuild
from paper_2609_38767_gb300 import synth

pytestmark = pytest.mark.gpu

TOL = {"f32": 1e-5, "bf16": 2e-2}


@pytest.fixture(scope="module")
def dev():
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    tbuild.build()
    tda.load()
    return torch.device("cuda:0")


def rel_fro(x, ref):
    x = np.asarray(x, dtype=np.float64)
    ref = np.asarray(ref, dtype=np.float64)
    return float(np.linalg.norm(x - ref) / max(np.linalg.norm(ref), 1e-300))


def make_factors(n, T, d_in, d_out, dtype, stream, sigma_b=0.1, mask_p=0.0, dist=0, e0=0, query=False):
    off = synth.QUERY_STREAM_OFFSET if query else 0
    ms = 1000 if query else 0
    A = synth.factors(synth.SEED_A, stream + off, n, T, d_in, 1.0, dist, e0, dtype, mask_p, mask_stream=ms)
    B = synth.factors(synth.SEED_B, stream + off, n, T, d_out, sigma_b, 0, e0, dtype, mask_p, mask_stream=ms)
    return A, B


def to_dev(x, dtype, device):
    if dtype == "bf16":
        return torch.from_numpy(x.view(np.int16)).view(torch.bfloat16).to(device)
    return torch.from_numpy(x).to(device)


TD = {"f32": tda.TDA_F32, "bf16": tda.TDA_BF16}


def gpu_project(L, dtype, A, B, N, route, device, ld=None, sign_ws=False):
    D = L.k_in * L.k_out
    ld = ld or D
    phi = torch.full((N, ld), float("nan"), dtype=torch.float32, device=device)
    ws, wsb = None, 0
    if route == tda.TDA_ROUTE_MATERIALIZE:
        wsb = tda.tda_workspace_size(tda.TDA_OP_PROJECT, L, TD[dtype], N, 0, route) * min(N, 3)
        ws = torch.empty(wsb, dtype=torch.uint8, device=device)
    elif sign_ws:  # the optional workspace of the factored route
        wsb = tda.tda_workspace_size(tda.TDA_OP_PROJECT, L, TD[dtype], N, 0, route)
        signs = 2 * L.k_in * (L.d_in + L.d_out) if L.k_in == 128 else 0
        assert wsb >= (signs + 255) // 256 * 256 + 2 * L.k_in * L.k_out * 4
        if sign_ws == "signs":  # room for the k = 128 sign tables only: whole examples per SM
            wsb = signs
        ws = torch.full((wsb,), 0x7F, dtype=torch.uint8, device=device)
    tda.tda_project(L, TD[dtype], A, B, N, phi, ld, route, ws, wsb)
    tda.tda_device_status()
    return phi[:, :D].cpu().numpy().reshape(N, L.k_out, L.k_in), phi


# ------------------------------------------------------------------ generator and signs
def test_device_generator_matches_numpy(dev):
    for dtype, dist, mask in [("f32", 0, 0.0), ("bf16", 0, 0.01), ("bf16", 1, 0.0), ("f32", 1, 0.05)]:
        n, T, d = 3, 37, 48
        ref = synth.factors(5, 7, n, T, d, 0.37, dist, 11, dtype, mask)
        out = torch.empty(n * T * d, dtype=torch.bfloat16 if dtype == "bf16" else torch.float32, device=dev)
        synth.fill_device(out, 5, 7, n, T, d, 0.37, dist, 11, mask)
        got = out.cpu()
        got = got.view(torch.int16).numpy().view(np.uint16) if dtype == "bf16" else got.numpy()
        np.testing.assert_array_equal(got.reshape(ref.shape), ref)


@pytest.mark.parametrize("rows,cols,side,layer", [(300, 48, 0, 0), (4096, 64, 1, 3), (130, 128, 0, 223),
                                                  (64, 16, 1, 7)])
def test_proj_entries_bit_exact(dev, orc, rows, cols, side, layer):
    out = torch.zeros(rows * cols, dtype=torch.int8, device=dev)
    tda.tda_proj_entries(12345, layer, side, 0, rows, cols, out)
    np.testing.assert_array_equal(out.cpu().numpy().reshape(rows, cols),
                                  orc.proj_entries(12345, layer, side, rows, cols))
    ident = torch.zeros(40 * 40, dtype=torch.int8, device=dev)
    tda.tda_proj_entries(0, 0, 0, 1, 40, 40, ident)
    np.testing.assert_array_equal(ident.cpu().numpy().reshape(40, 40), np.eye(40, dtype=np.int8))


# ------------------------------------------------------------------ projection
PROJ_CASES = [
    # (N, T, d_in, d_out, k_in, k_out, dtype, kind)
    (64, 32, 256, 256, 16, 16, "f32", 0),        # the 256x256 fp32 layer, k = 16
    (5, 45, 200, 136, 32, 48, "bf16", 0),        # ragged T, d and k
    (3, 130, 512, 1024, 32, 32, "bf16", 0),      # T over one 128-token tile
    (4, 19, 96, 160, 80, 72, "f32", 0),          # k over one 64-wide tile
    (2, 7, 24, 16, 24, 16, "f32", 1),            # identity map: Phi = DW
    (3, 64, 256, 512, 128, 64, "bf16", 0),       # wide k
    (2, 257, 128, 128, 64, 64, "bf16", 0),       # tokens spanning 3 tiles
]


@pytest.mark.parametrize("case", PROJ_CASES)
@pytest.mark.parametrize("route", [tda.TDA_ROUTE_FACTORED, tda.TDA_ROUTE_MATERIALIZE])
def test_project_matches_oracle(dev, orc, case, route):
    N, T, di, do, ki, ko, dtype, kind = case
    A, B = make_factors(N, T, di, do, dtype, stream=3, mask_p=0.02)
    L = tda.LayerDesc(di, do, T, ki, ko, seed=99, layer=5, kind=kind)
    got, _ = gpu_project(L, dtype, to_dev(A, dtype, dev), to_dev(B, dtype, dev), N, route, dev)
    ref = orc.project(synth.to_f64(A, dtype), synth.to_f64(B, dtype), ki, ko, 99, 5, kind)
    err = rel_fro(got, ref)
    assert err <= TOL[dtype], err
    for n in range(N):  # per example as well
        assert rel_fro(got[n], ref[n]) <= TOL[dtype]


def test_project_leading_dimension_and_edge_sizes(dev, orc):
    N, T, di, do, ki, ko = 4, 20, 64, 32, 16, 8
    A, B = make_factors(N, T, di, do, "f32", stream=4)
    L = tda.LayerDesc(di, do, T, ki, ko, seed=1, layer=2)
    got, phi = gpu_project(L, "f32", to_dev(A, "f32", dev), to_dev(B, "f32", dev), N,
                           tda.TDA_ROUTE_FACTORED, dev, ld=200)
    assert torch.isnan(phi[:, ki * ko:]).all()  # untouched padding
    ref = orc.project(synth.to_f64(A, "f32"), synth.to_f64(B, "f32"), ki, ko, 1, 2)
    assert rel_fro(got, ref) <= 1e-5
    # T = 0: DW = 0; N = 0: nothing to do
    L0 = tda.LayerDesc(di, do, 0, ki, ko)
    phi0 = torch.full((3, ki * ko), 7.0, device=dev)
    tda.tda_project(L0, tda.TDA_F32, None, None, 3, phi0, ki * ko)
    assert (phi0 == 0).all()
    tda.tda_project(L, tda.TDA_F32, None, None, 0, None, ki * ko)
    tda.tda_device_status()


# ------------------------------------------------------------------ exact similarity
@pytest.mark.parametrize("dtype", ["f32", "bf16"])
@pytest.mark.parametrize("route", [tda.TDA_ROUTE_GRAM, tda.TDA_ROUTE_MATERIALIZE, tda.TDA_ROUTE_AUTO])
# 2nd, 3rd: split-K Frobenius dots (3rd: a ragged last feature slice)
@pytest.mark.parametrize("shape", [(3, 5, 21, 40, 24), (3, 5, 7, 256, 264), (2, 11, 5, 264, 136)])
def test_similarity_exact_matches_oracle(dev, orc, dtype, route, shape):
    nq, nt, T, di, do = shape
    Aq, Bq = make_factors(nq, T, di, do, dtype, stream=6, query=True)
    At, Bt = make_factors(nt, T, di, do, dtype, stream=6)
    L = tda.LayerDesc(di, do, T, 1, 1)
    S = torch.full((nq, nt + 3), 0.5, device=dev)
    wsb = tda.tda_workspace_size(tda.TDA_OP_SIMILARITY_EXACT, L, TD[dtype], nq, nt, route) * 2
    ws = torch.empty(max(wsb, 1), dtype=torch.uint8, device=dev)
    tda.tda_similarity_exact(L, TD[dtype], to_dev(Aq, dtype, dev), to_dev(Bq, dtype, dev), nq,
                             to_dev(At, dtype, dev), to_dev(Bt, dtype, dev), nt, S, nt + 3, 1.0, route,
                             ws, wsb)
    tda.tda_device_status()
    ref = orc.similarity(synth.to_f64(Aq, dtype), synth.to_f64(Bq, dtype), synth.to_f64(At, dtype),
                         synth.to_f64(Bt, dtype)) + 0.5
    assert rel_fro(S[:, :nt].cpu().numpy(), ref) <= TOL[dtype]
    assert (S[:, nt:] == 0.5).all()


# ------------------------------------------------------------------ preconditioned scores
def _precond_pipeline(dev, orc, N, Nq, T, di, do, k, dtype, sdt, lam_abs, lam_rel, mask_p=0.0):
    A, B = make_factors(N, T, di, do, dtype, stream=8, mask_p=mask_p)
    Aq, Bq = make_factors(Nq, T, di, do, dtype, stream=8, mask_p=mask_p, query=True)
    L = tda.LayerDesc(di, do, T, k, k, seed=0, layer=0)
    D = k * k
    _, phi = gpu_project(L, dtype, to_dev(A, dtype, dev), to_dev(B, dtype, dev), N, tda.TDA_ROUTE_FACTORED, dev)
    _, q = gpu_project(L, dtype, to_dev(Aq, dtype, dev), to_dev(Bq, dtype, dev), Nq, tda.TDA_ROUTE_FACTORED, dev)
    state = torch.empty(tda.tda_precondition_state_bytes(D, sdt), dtype=torch.uint8, device=dev)
    tda.tda_precondition(tda.TDA_PC_RESET, 1, D, sdt, state)
    half = N // 2  # two streamed chunks
    tda.tda_precondition(tda.TDA_PC_FIT_ACCUM, 1, D, sdt, state, phi=phi, n=half, ld_phi=D)
    tda.tda_precondition(tda.TDA_PC_FIT_ACCUM, 1, D, sdt, state, phi=phi[half:], n=N - half, ld_phi=D)
    tda.tda_precondition(tda.TDA_PC_FACTOR, 1, D, sdt, state, n_total=N, lambda_abs=lam_abs,
                         lambda_rel_mean_eig=lam_rel)
    qhat = torch.empty((Nq, D), dtype=torch.float64 if sdt == tda.TDA_F64 else torch.float32, device=dev)
    tda.tda_precondition(tda.TDA_PC_APPLY, 1, D, sdt, state, q=q, n_q=Nq, ld_q=D, qhat=qhat, ld_qhat=D)
    S = torch.empty((Nq, N), device=dev)
    tda.tda_score(qhat, sdt, Nq, D, phi, N, D, D, S, N)
    info = tda.tda_precondition_info(1, D, sdt, state)
    tda.tda_device_status()
    # oracle, end to end from the same input bits
    fo = orc.project(synth.to_f64(A, dtype), synth.to_f64(B, dtype), k, k, 0, 0).reshape(N, D)
    fq = orc.project(synth.to_f64(Aq, dtype), synth.to_f64(Bq, dtype), k, k, 0, 0).reshape(Nq, D)
    F = orc.fisher(fo)
    lam = orc.damping(F, lam_abs, lam_rel)
    Sref = orc.score(orc.precondition(F, lam, fq), fo)
    return S.cpu().numpy(), Sref, info, lam


def test_preconditioned_scores_fp32_layer_fp64_state(dev, orc):
    # d 256 -> 256, fp32, T = 32, 64 train / 8 query, k = 16, lambda = 1e-3
    S, Sref, info, lam = _precond_pipeline(dev, orc, 64, 8, 32, 256, 256, 16, "f32", tda.TDA_F64, 1e-3, 0.0)
    assert abs(info[0] - lam) <= 1e-12 * lam and info[2] == 0 and info[3] == 64
    assert rel_fro(S, Sref) <= 1e-5


def test_preconditioned_scores_bf16_fp32_state_relative_damping(dev, orc):
    S, Sref, info, lam = _precond_pipeline(dev, orc, 96, 16, 40, 128, 192, 16, "bf16", tda.TDA_F32,
                                           0.0, 1e-2, mask_p=0.01)
    assert abs(info[0] - lam) <= 1e-5 * lam
    assert rel_fro(S, Sref) <= 2e-2


@pytest.mark.parametrize("D", [8, 64, 96])  # 64, 96: the one-launch cluster factorisation
def test_precondition_not_spd_is_reported(dev, D):
    state = torch.empty(tda.tda_precondition_state_bytes(D, tda.TDA_F32), dtype=torch.uint8, device=dev)
    tda.tda_precondition(tda.TDA_PC_RESET, 1, D, tda.TDA_F32, state)
    phi = torch.ones((2, D), device=dev)
    tda.tda_precondition(tda.TDA_PC_FIT_ACCUM, 1, D, tda.TDA_F32, state, phi=phi, n=2, ld_phi=D)
    # make the accumulated matrix indefinite by hand
    m = state[64:64 + 4 * D * D].view(torch.float32).view(D, D)
    m[3, 3] = -100.0
    tda.tda_precondition(tda.TDA_PC_FACTOR, 1, D, tda.TDA_F32, state, n_total=2, lambda_abs=1e-3)
    with pytest.raises(tda.TdaError) as e:
        tda.tda_precondition_info(1, D, tda.TDA_F32, state)
    assert e.value.status == tda.TDA_ERR_NOT_SPD
    q = torch.ones((1, D), device=dev)
    qh = torch.zeros((1, D), device=dev)
    tda.tda_precondition(tda.TDA_PC_APPLY, 1, D, tda.TDA_F32, state, q=q, n_q=1, ld_q=D, qhat=qh, ld_qhat=D)
    assert torch.isnan(qh).all()


# ------------------------------------------------------------------ score and top-k
@pytest.mark.parametrize("qdt", [tda.TDA_F32, tda.TDA_F64])
def test_score_and_accumulate(dev, orc, qdt):
    rng = np.random.default_rng(0)
    nq, nt, D = 70, 133, 1029
    Q = rng.standard_normal((nq, D)).astype(np.float32)
    P = rng.standard_normal((nt, D)).astype(np.float32)
    Qd = torch.from_numpy(Q).to(dev).to(torch.float64 if qdt == tda.TDA_F64 else torch.float32)
    S = torch.full((nq, nt), 2.0, device=dev)
    tda.tda_score(Qd, qdt, nq, D, torch.from_numpy(P).to(dev), nt, D, D, S, nt, beta=1.0)
    tda.tda_device_status()
    ref = orc.score(Q, P) + 2.0
    assert rel_fro(S.cpu().numpy(), ref) <= 1e-5


def test_topk_selection_bit_exact_on_gpu_scores(dev, orc):
    rng = np.random.default_rng(1)
    nq, nt, k = 9, 5000, 100
    S = (np.round(rng.standard_normal((nq, nt)) * 64) / 64).astype(np.float32)  # many ties
    S[0, :] = 0.0
    S[1, 17] = -0.0
    Sd = torch.from_numpy(S).to(dev)
    idx = torch.empty((nq, k), dtype=torch.int32, device=dev)
    val = torch.empty((nq, k), device=dev)
    tda.tda_topk(Sd, nq, nt, nt, k, idx, val)
    tda.tda_device_status()
    oi, ov = orc.topk(S.astype(np.float64), k)
    np.testing.assert_array_equal(idx.cpu().numpy(), oi)
    np.testing.assert_array_equal(val.cpu().numpy(), ov.astype(np.float32))


def test_topk_nan_first_and_signed_zeros(dev, orc):
    # NaN ranks above every number (NaNs by index), -0 ties with +0 (by index): the GPU and the
    # oracle's total order agree on every index, values compared bit for bit apart from NaN payloads
    rng = np.random.default_rng(11)
    nq, nt, k = 4, 3000, 60
    S = (np.round(rng.standard_normal((nq, nt)) * 8) / 8).astype(np.float32)
    S[0, [5, 900, 2999]] = np.nan
    S[1, :] = 0.0
    S[1, ::3] = -0.0
    S[2, [10, 20]] = np.inf
    S[2, [30, 40]] = np.nan
    S[3, :] = -np.inf
    S[3, 100:140] = np.nan
    idx = torch.empty((nq, k), dtype=torch.int32, device=dev)
    val = torch.empty((nq, k), device=dev)
    tda.tda_topk(torch.from_numpy(S).to(dev), nq, nt, nt, k, idx, val)
    tda.tda_device_status()
    oi, ov = orc.topk(S.astype(np.float64), k)
    np.testing.assert_array_equal(idx.cpu().numpy(), oi)
    np.testing.assert_array_equal(val.cpu().numpy(), ov.astype(np.float32))
    assert list(oi[0, :3]) == [5, 900, 2999] and list(oi[2, :4]) == [30, 40, 10, 20]
    g = val.cpu().numpy()
    assert (np.signbit(g[1]) == np.signbit(S[1, oi[1]])).all()  # each selected zero keeps its sign


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_config1_layer_three_routes_agree(dev, orc, dtype):
    # the 256 x 256 layer, T = 32, k = 16, 8 queries x 64 train: projected similarity by the
    # factored, materialised and Gram routes against the oracle, and the exact (unprojected)
    # similarity by the materialised and Gram routes
    nq, nt, T, d, k = 8, 64, 32, 256, 16
    Aq, Bq = make_factors(nq, T, d, d, dtype, stream=0, query=True)
    At, Bt = make_factors(nt, T, d, d, dtype, stream=0)
    L = tda.LayerDesc(d, d, T, k, k, seed=0, layer=0)
    args = [to_dev(x, dtype, dev) for x in (Aq, Bq, At, Bt)]
    fq = orc.project(synth.to_f64(Aq, dtype), synth.to_f64(Bq, dtype), k, k, 0, 0)
    ft = orc.project(synth.to_f64(At, dtype), synth.to_f64(Bt, dtype), k, k, 0, 0)
    ref_p = orc.score(fq, ft)
    ref_x = orc.similarity(*(synth.to_f64(x, dtype) for x in (Aq, Bq, At, Bt)))
    got = {}
    for route in (tda.TDA_ROUTE_FACTORED, tda.TDA_ROUTE_MATERIALIZE, tda.TDA_ROUTE_GRAM):
        wsb = max(tda.tda_workspace_size(tda.TDA_OP_SIMILARITY_PROJECTED, L, TD[dtype], nq, nt, route), 256)
        ws = torch.empty(wsb, dtype=torch.uint8, device=dev)
        S = torch.empty((nq, nt), device=dev)
        tda.tda_similarity_projected(L, TD[dtype], args[0], args[1], nq, args[2], args[3], nt, S, nt, 0.0, route,
                                     ws, wsb)
        tda.tda_device_status()
        got[route] = S.cpu().numpy()
        assert rel_fro(got[route], ref_p) <= TOL[dtype], route
    for route in (tda.TDA_ROUTE_MATERIALIZE, tda.TDA_ROUTE_GRAM):
        wsb = max(tda.tda_workspace_size(tda.TDA_OP_SIMILARITY_EXACT, L, TD[dtype], nq, nt, route), 256)
        ws = torch.empty(wsb, dtype=torch.uint8, device=dev)
        S = torch.empty((nq, nt), device=dev)
        tda.tda_similarity_exact(L, TD[dtype], args[0], args[1], nq, args[2], args[3], nt, S, nt, 0.0, route, ws,
                                 wsb)
        tda.tda_device_status()
        assert rel_fro(S.cpu().numpy(), ref_x) <= TOL[dtype], route


@pytest.mark.parametrize("k", [1, 7, 1024])
def test_topk_sizes(dev, orc, k):
    rng = np.random.default_rng(k)
    nq, nt = 3, 1500
    S = rng.standard_normal((nq, nt)).astype(np.float32)
    idx = torch.empty((nq, k), dtype=torch.int32, device=dev)
    tda.tda_topk(torch.from_numpy(S).to(dev), nq, nt, nt, k, idx, None)
    oi, _ = orc.topk(S.astype(np.float64), k)
    np.testing.assert_array_equal(idx.cpu().numpy(), oi)


def test_route_auto_and_calibration(dev, orc):
    ws = torch.empty(tda.TDA_CALIBRATE_WS_BYTES, dtype=torch.uint8, device=dev)
    rates = tda.tda_route_calibrate(ws, tda.TDA_CALIBRATE_WS_BYTES)
    assert all(r > 0 for r in rates), rates
    L = tda.LayerDesc(2048, 2048, 512, 32, 32)
    chosen, cost = tda.tda_route(L, tda.TDA_OP_PROJECT, 4096, 0, tda.TDA_BF16)
    assert chosen == tda.TDA_ROUTE_FACTORED and cost[0] < cost[1]
    tda.tda_route_set_model(0)
    chosen, cost = tda.tda_route(L, tda.TDA_OP_SIMILARITY_EXACT, 1, 8, tda.TDA_BF16)
    assert chosen == orc.route_costs(2, 1, 8, 512, 2048, 2048)[0]


# ------------------------------------------------------------------ tensor-core projection specifics
@pytest.mark.parametrize("k,sign_ws", [(32, False), (32, True), (128, False), (128, "signs"), (128, True)])
def test_tc_projection_signs_bit_exact(dev, orc, k, sign_ws):
    # One-hot factors: A_n = I (T = d_in tokens), B_n = e_r at token t only, so
    # Phi_n / scale = outer(S_out[r, :], S_in[t, :]) exactly -- the signs the
    # tensor-core kernel generated on chip, compared bit for bit with the oracle's.
    d, N = 128, 4
    picks = [(0, 5), (77, 127), (127, 64), (31, 0)]  # (t, r) per example
    A = np.zeros((N, d, d), dtype=np.float32)
    B = np.zeros((N, d, d), dtype=np.float32)
    for n, (t, r) in enumerate(picks):
        A[n] = np.eye(d, dtype=np.float32)
        B[n, t, r] = 1.0
    Ab = torch.from_numpy(A).to(dev).to(torch.bfloat16)
    Bb = torch.from_numpy(B).to(dev).to(torch.bfloat16)
    L = tda.LayerDesc(d, d, d, k, k, seed=2024, layer=9)
    assert tda.tda_project_engine(L, tda.TDA_BF16, Ab, Bb) == 1
    got, _ = gpu_project(L, "bf16", Ab, Bb, N, tda.TDA_ROUTE_FACTORED, dev, sign_ws=sign_ws)
    S_in = orc.proj_entries(2024, 9, 0, d, k).astype(np.float32)
    S_out = orc.proj_entries(2024, 9, 1, d, k).astype(np.float32)
    for n, (t, r) in enumerate(picks):
        np.testing.assert_array_equal(got[n] * k, np.outer(S_out[r], S_in[t]))


TC_CASES = [
    # (N, T, d_in, d_out, k, dtype): persistent loop, ragged K chunks, T = 1, T over tiles
    (400, 200, 64, 72, 16, "bf16"),
    (7, 1, 136, 200, 32, "bf16"),
    (5, 129, 136, 64, 64, "bf16"),
    (3, 384, 1024, 256, 32, "bf16"),
    (160, 16, 2048, 2048, 32, "bf16"),
    # fewer examples than SMs: clusters of CTAs split an example's token tiles
    (2, 1024, 256, 512, 32, "bf16"),    # 4-CTA clusters, 2 tiles per CTA
    (50, 300, 128, 64, 16, "bf16"),     # 4-CTA clusters; more clusters than fit
    (64, 512, 512, 256, 64, "bf16"),    # 2-CTA clusters (the query batch shape)
    (1, 384, 64, 64, 32, "bf16"),       # one example over 2 CTAs, uneven tiles
    # two token tiles per pipeline stage (many units): groups that straddle examples
    (250, 300, 64, 72, 32, "bf16"),
    (700, 256, 64, 128, 64, "bf16"),
    # at least one example per SM: 32 token rows staged at a time, groups straddling examples
    (300, 300, 200, 136, 64, "bf16"),
    (160, 48, 64, 64, 128, "bf16"),
    # short sequences packed several examples to a tile, ragged last tile
    (2001, 48, 64, 64, 16, "bf16"),     # 2 per tile, 32 rows unused, one tile per stage pair
    (20001, 8, 64, 64, 16, "bf16"),     # 16 per tile
    (300, 3, 128, 64, 32, "bf16"),      # 42 per tile
    (1000, 64, 256, 128, 64, "bf16"),   # 2 per tile, K = 64
    # k = 128: one tile per stage, the epilogue contracts 64-token halves
    (200, 200, 136, 200, 128, "bf16"),  # persistent loop, ragged K chunks and last tile
    (5, 384, 256, 128, 128, "bf16"),    # fewer examples than SMs: 2-CTA clusters
    (1, 200, 64, 64, 128, "bf16"),      # one example over 2 CTAs, ragged second tile
    (40, 48, 64, 64, 128, "bf16"),      # short sequences stay one example per tile
    (3, 1, 72, 64, 128, "bf16"),        # T = 1
]


@pytest.mark.parametrize("case", [c for c in TC_CASES if c[4] == 128] + [(9, 130, 1000, 2056, 128, "bf16")])
def test_tc_projection_k128_sign_tables_match_oracle(dev, orc, case):
    # k = 128 with the optional workspace: both sides' sign tables written once per call and
    # read by TMA beside the factor tiles (d not a multiple of 64: zero-filled last chunk)
    N, T, di, do, k, dtype = case
    A, B = make_factors(N, T, di, do, dtype, stream=12, sigma_b=0.03, mask_p=0.01)
    L = tda.LayerDesc(di, do, T, k, k, seed=6, layer=4)
    Ad, Bd = to_dev(A, dtype, dev), to_dev(B, dtype, dev)
    got, _ = gpu_project(L, dtype, Ad, Bd, N, tda.TDA_ROUTE_FACTORED, dev, sign_ws="signs")
    plain, _ = gpu_project(L, dtype, Ad, Bd, N, tda.TDA_ROUTE_FACTORED, dev)
    np.testing.assert_array_equal(got, plain)  # same signs, same arithmetic order
    ref = orc.project(synth.to_f64(A, dtype), synth.to_f64(B, dtype), k, k, 6, 4)
    assert max(rel_fro(got[n], ref[n]) for n in range(N)) <= TOL[dtype]
    # the whole workspace: sign tables and balanced token-tile ranges
    bal, _ = gpu_project(L, dtype, Ad, Bd, N, tda.TDA_ROUTE_FACTORED, dev, sign_ws=True)
    assert max(rel_fro(bal[n], ref[n]) for n in range(N)) <= TOL[dtype]


@pytest.mark.parametrize("ws", [False, True])
@pytest.mark.parametrize("case", TC_CASES)
def test_tc_projection_matches_oracle(dev, orc, case, ws):
    # ws: with the optional workspace every SM takes an equal run of token tiles (examples split
    # between SMs are summed from partial blocks); without it, whole examples or clusters
    N, T, di, do, k, dtype = case
    A, B = make_factors(N, T, di, do, dtype, stream=11, sigma_b=0.03, mask_p=0.01)
    L = tda.LayerDesc(di, do, T, k, k, seed=5, layer=3)
    Ad, Bd = to_dev(A, dtype, dev), to_dev(B, dtype, dev)
    assert tda.tda_project_engine(L, TD[dtype], Ad, Bd) == 1  # the tensor-core kernel runs
    got, _ = gpu_project(L, dtype, Ad, Bd, N, tda.TDA_ROUTE_FACTORED, dev, sign_ws=ws)
    ref = orc.project(synth.to_f64(A, dtype), synth.to_f64(B, dtype), k, k, 5, 3)
    assert rel_fro(got, ref) <= TOL[dtype]
    worst = max(rel_fro(got[n], ref[n]) for n in range(N))
    assert worst <= TOL[dtype], worst


BAL_CASES = [
    # (N, T, d_in, d_out, k): examples split over several SMs, few examples, one tile per example
    (1, 2048, 128, 64, 128),    # one example over 16 SMs
    (5, 2048, 136, 200, 64),    # 80 tiles: some SMs idle (grid = tiles)
    (16, 2048, 256, 128, 128),  # 256 tiles over every SM, split examples at most boundaries
    (153, 1024, 64, 72, 32),    # 1224 tiles: ranges of 8 or 9 tiles, G = 2 groups across examples
    (200, 100, 64, 64, 16),     # one tile per example: nothing split
    (7, 300, 64, 64, 64),       # 21 tiles, ragged last tile of every example
]


@pytest.mark.parametrize("case", BAL_CASES)
def test_tc_projection_balanced_ranges(dev, orc, case):
    # Balanced ranges are deterministic (the split examples' partial blocks are added in SM
    # order whichever SM finishes last) and leave the workspace's counters clear: a second call
    # on the same workspace reproduces the first bit for bit; both match the oracle.
    N, T, di, do, k = case
    A, B = make_factors(N, T, di, do, "bf16", stream=13, sigma_b=0.03, mask_p=0.01)
    L = tda.LayerDesc(di, do, T, k, k, seed=8, layer=2)
    Ad, Bd = to_dev(A, "bf16", dev), to_dev(B, "bf16", dev)
    wsb = tda.tda_workspace_size(tda.TDA_OP_PROJECT, L, tda.TDA_BF16, N, 0, tda.TDA_ROUTE_FACTORED)
    ws = torch.full((wsb,), 0x5A, dtype=torch.uint8, device=dev)
    outs = []
    for _ in range(2):
        phi = torch.full((N, k * k), float("nan"), device=dev)
        tda.tda_project(L, tda.TDA_BF16, Ad, Bd, N, phi, k * k, tda.TDA_ROUTE_FACTORED, ws, wsb)
        tda.tda_device_status()
        outs.append(phi.cpu().numpy().reshape(N, k, k))
    np.testing.assert_array_equal(outs[0], outs[1])
    ref = orc.project(synth.to_f64(A, "bf16"), synth.to_f64(B, "bf16"), k, k, 8, 2)
    worst = max(rel_fro(outs[0][n], ref[n]) for n in range(N))
    assert worst <= TOL["bf16"], worst


@pytest.mark.parametrize("sdt,D,lam_abs,lam_rel,tol", [(tda.TDA_F64, 70, 1e-3, 0.0, 1e-9),
                                                       (tda.TDA_F32, 96, 0.0, 1e-2, 1e-4),
                                                       (tda.TDA_F32, 1000, 0.0, 1e-2, 1e-3),
                                                       (tda.TDA_F32, 1024, 0.0, 1e-2, 1e-3)])
def test_precondition_batched_layers_match_oracle(dev, orc, sdt, D, lam_abs, lam_rel, tol):
    # three layers side by side in each feature row, ragged D, streamed in two chunks
    rng = np.random.default_rng(D)
    nl, N, Nq = 3, 150, 11
    phi = (rng.standard_normal((N, nl * D)) * rng.uniform(0.5, 2.0, nl * D)).astype(np.float32)
    q = rng.standard_normal((Nq, nl * D)).astype(np.float32)
    per = tda.tda_precondition_state_bytes(D, sdt)
    state = torch.empty(nl * per, dtype=torch.uint8, device=dev)
    phid, qd = torch.from_numpy(phi).to(dev), torch.from_numpy(q).to(dev)
    tda.tda_precondition(tda.TDA_PC_RESET, nl, D, sdt, state)
    tda.tda_precondition(tda.TDA_PC_FIT_ACCUM, nl, D, sdt, state, phi=phid, n=70, ld_phi=nl * D)
    tda.tda_precondition(tda.TDA_PC_FIT_ACCUM, nl, D, sdt, state, phi=phid[70:], n=N - 70, ld_phi=nl * D)
    tda.tda_precondition(tda.TDA_PC_FACTOR, nl, D, sdt, state, n_total=N, lambda_abs=lam_abs,
                         lambda_rel_mean_eig=lam_rel)
    qh = torch.empty((Nq, nl * D), dtype=torch.float64 if sdt == tda.TDA_F64 else torch.float32, device=dev)
    tda.tda_precondition(tda.TDA_PC_APPLY, nl, D, sdt, state, q=qd, n_q=Nq, ld_q=nl * D, qhat=qh, ld_qhat=nl * D)
    info = tda.tda_precondition_info(nl, D, sdt, state)
    tda.tda_device_status()
    got = qh.cpu().numpy().astype(np.float64)
    for l in range(nl):
        F = orc.fisher(phi[:, l * D:(l + 1) * D].astype(np.float64))
        lam = orc.damping(F, lam_abs, lam_rel)
        assert abs(info[4 * l] - lam) <= 1e-5 * lam and info[4 * l + 2] == 0
        ref = orc.precondition(F, lam, q[:, l * D:(l + 1) * D].astype(np.float64))
        assert rel_fro(got[:, l * D:(l + 1) * D], ref) <= tol


@pytest.mark.parametrize("D,nl,chunks,pad", [(128, 1, (5, 40), 0), (1000, 3, (70, 80, 31), 4),
                                             (1024, 2, (4096,), 0), (256, 2, (1, 33, 64), 8)])
def test_fisher_fit_accumulates_phi_t_phi(dev, orc, D, nl, chunks, pad):
    # FIT_ACCUM on an fp32 state (the tensor-core fit for D >= 128): M_l = sum over the streamed
    # chunks of Phi_l^T Phi_l, compared on the lower triangle with the oracle's Fisher times N.
    # Ragged D makes a layer's last tile read the next layer's features (rows past D, discarded);
    # chunks of 1, 5, 31, 33 examples end inside a 32-example operand chunk; 4096 examples wrap
    # every pipeline ring many times.
    rng = np.random.default_rng(D + nl)
    N = sum(chunks)
    W = nl * D + pad
    phi = (rng.standard_normal((N, W)) * rng.uniform(0.5, 2.0, W)).astype(np.float32)
    sdt = tda.TDA_F32
    per = tda.tda_precondition_state_bytes(D, sdt)
    state = torch.empty(nl * per, dtype=torch.uint8, device=dev)
    phid = torch.from_numpy(phi).to(dev)
    tda.tda_precondition(tda.TDA_PC_RESET, nl, D, sdt, state)
    e0 = 0
    for c in chunks:
        tda.tda_precondition(tda.TDA_PC_FIT_ACCUM, nl, D, sdt, state, phi=phid[e0:], n=c, ld_phi=W)
        e0 += c
    tda.tda_device_status()
    low = np.tril_indices(D)
    for l in range(nl):
        M = state[l * per + 64:l * per + 64 + 4 * D * D].view(torch.float32).view(D, D).cpu().numpy()
        ref = N * orc.fisher(phi[:, l * D:(l + 1) * D].astype(np.float64))
        assert np.isfinite(M[low]).all()
        assert rel_fro(M[low], ref[low]) <= 1e-5
        # element by element against the Cauchy-Schwarz scale of each entry
        scale = np.sqrt(np.outer(np.diag(ref), np.diag(ref)))
        assert (np.abs(M - ref)[low] <= 1e-5 * scale[low]).all()


@pytest.mark.parametrize("D,Nq,nl", [(64, 11, 1), (96, 70, 3), (1024, 64, 2), (1000, 9, 1), (128, 300, 1)])
def test_precondition_factor_apply_matches_oracle(dev, orc, D, Nq, nl):
    # FACTOR_APPLY: one launch for an fp32 state with D a multiple of 32 and <= 256 queries (the
    # queries solved alongside the factorisation), FACTOR then APPLY otherwise (D = 1000, 300 queries)
    rng = np.random.default_rng(D + Nq)
    N = 150
    phi = (rng.standard_normal((N, nl * D)) * rng.uniform(0.5, 2.0, nl * D)).astype(np.float32)
    q = rng.standard_normal((Nq, nl * D + 3)).astype(np.float32)
    sdt = tda.TDA_F32
    per = tda.tda_precondition_state_bytes(D, sdt)
    state = torch.empty(nl * per, dtype=torch.uint8, device=dev)
    phid, qd = torch.from_numpy(phi).to(dev), torch.from_numpy(q).to(dev)
    tda.tda_precondition(tda.TDA_PC_RESET, nl, D, sdt, state)
    tda.tda_precondition(tda.TDA_PC_FIT_ACCUM, nl, D, sdt, state, phi=phid, n=N, ld_phi=nl * D)
    qh = torch.full((Nq, nl * D + 5), 7.0, device=dev)
    tda.tda_precondition(tda.TDA_PC_FACTOR_APPLY, nl, D, sdt, state, n_total=N, lambda_abs=0.0,
                         lambda_rel_mean_eig=1e-2, q=qd, n_q=Nq, ld_q=nl * D + 3, qhat=qh, ld_qhat=nl * D + 5)
    info = tda.tda_precondition_info(nl, D, sdt, state)
    tda.tda_device_status()
    got = qh.cpu().numpy().astype(np.float64)
    assert (got[:, nl * D:] == 7.0).all()
    for l in range(nl):
        F = orc.fisher(phi[:, l * D:(l + 1) * D].astype(np.float64))
        lam = orc.damping(F, 0.0, 1e-2)
        assert abs(info[4 * l] - lam) <= 1e-5 * lam and info[4 * l + 2] == 0
        ref = orc.precondition(F, lam, q[:, l * D:(l + 1) * D].astype(np.float64))
        assert rel_fro(got[:, l * D:(l + 1) * D], ref) <= 1e-3
    # the same state applied again through APPLY gives the same rows (up to summation order)
    qh2 = torch.empty((Nq, nl * D), device=dev)
    tda.tda_precondition(tda.TDA_PC_APPLY, nl, D, sdt, state, q=qd, n_q=Nq, ld_q=nl * D + 3, qhat=qh2, ld_qhat=nl * D)
    tda.tda_device_status()
    assert rel_fro(qh2.cpu().numpy(), got[:, :nl * D]) <= 1e-5


@pytest.mark.parametrize("D,nl,N,Nq,op", [(2048, 2, 700, 37, "split"), (2048, 1, 3000, 300, "fused"),
                                          (4096, 2, 400, 5, "fused"), (2048, 3, 150, 130, "inplace")])
def test_precondition_blocked_matches_oracle(dev, orc, D, nl, N, Nq, op):
    # fp32 state, D a multiple of 128 and >= 2048: 128-column panels, tensor-core trailing updates
    # and substitutions. Ragged query counts (not multiples of the 128-row tiles), N above and
    # below D (the oracle solves through the D x D Cholesky or its Woodbury form), the two ops
    # split (FACTOR, then APPLY with padded row strides), fused, or solved in place (qhat = q).
    orc.set_threads(os.cpu_count() or 1)
    rng = np.random.default_rng(D + N + Nq)
    phi = (rng.standard_normal((N, nl * D)) * rng.uniform(0.5, 2.0, nl * D)).astype(np.float32)
    ldq = nl * D + (4 if op == "split" else 0)
    q = rng.standard_normal((Nq, ldq)).astype(np.float32)
    sdt = tda.TDA_F32
    per = tda.tda_precondition_state_bytes(D, sdt)
    state = torch.empty(nl * per, dtype=torch.uint8, device=dev)
    phid, qd = torch.from_numpy(phi).to(dev), torch.from_numpy(q).to(dev)
    tda.tda_precondition(tda.TDA_PC_RESET, nl, D, sdt, state)
    tda.tda_precondition(tda.TDA_PC_FIT_ACCUM, nl, D, sdt, state, phi=phid, n=N, ld_phi=nl * D)
    if op == "inplace":
        qh, ldh = qd, ldq
    else:
        ldh = nl * D + (8 if op == "split" else 0)
        qh = torch.full((Nq, ldh), 7.0, device=dev)
    if op == "split":
        tda.tda_precondition(tda.TDA_PC_FACTOR, nl, D, sdt, state, n_total=N, lambda_rel_mean_eig=1e-2)
        tda.tda_precondition(tda.TDA_PC_APPLY, nl, D, sdt, state, q=qd, n_q=Nq, ld_q=ldq, qhat=qh, ld_qhat=ldh)
    else:
        tda.tda_precondition(tda.TDA_PC_FACTOR_APPLY, nl, D, sdt, state, n_total=N, lambda_rel_mean_eig=1e-2,
                             q=qd, n_q=Nq, ld_q=ldq, qhat=qh, ld_qhat=ldh)
    info = tda.tda_precondition_info(nl, D, sdt, state)
    tda.tda_device_status()
    got = qh.cpu().numpy().astype(np.float64)
    if op == "split":
        assert (got[:, nl * D:] == 7.0).all()
    for l in range(nl):
        P = phi[:, l * D:(l + 1) * D].astype(np.float64)
        lam = orc.damping_features(P, 0.0, 1e-2)
        assert abs(info[4 * l] - lam) <= 1e-5 * lam and info[4 * l + 2] == 0
        Ql = q[:, l * D:(l + 1) * D].astype(np.float64)
        ref = orc.precondition(orc.fisher(P), lam, Ql) if N >= D else orc.precondition_lowrank(P, lam, Ql)
        assert rel_fro(got[:, l * D:(l + 1) * D], ref) <= 1e-3, l


def test_precondition_blocked_not_spd_gives_nan(dev):
    D = 2048
    state = torch.empty(tda.tda_precondition_state_bytes(D, tda.TDA_F32), dtype=torch.uint8, device=dev)
    tda.tda_precondition(tda.TDA_PC_RESET, 1, D, tda.TDA_F32, state)
    phi = torch.ones((2, D), device=dev)
    tda.tda_precondition(tda.TDA_PC_FIT_ACCUM, 1, D, tda.TDA_F32, state, phi=phi, n=2, ld_phi=D)
    m = state[64:64 + 4 * D * D].view(torch.float32).view(D, D)
    m[1500, 1500] = -1e6
    q = torch.ones((3, D), device=dev)
    qh = torch.zeros((3, D), device=dev)
    tda.tda_precondition(tda.TDA_PC_FACTOR_APPLY, 1, D, tda.TDA_F32, state, n_total=2, lambda_abs=1e-3,
                         q=q, n_q=3, ld_q=D, qhat=qh, ld_qhat=D)
    with pytest.raises(tda.TdaError) as e:
        tda.tda_precondition_info(1, D, tda.TDA_F32, state)
    assert e.value.status == tda.TDA_ERR_NOT_SPD
    assert torch.isnan(qh).all()


@pytest.mark.parametrize("D", [64, 8])
def test_precondition_factor_apply_not_spd_gives_nan(dev, D):
    state = torch.empty(tda.tda_precondition_state_bytes(D, tda.TDA_F32), dtype=torch.uint8, device=dev)
    tda.tda_precondition(tda.TDA_PC_RESET, 1, D, tda.TDA_F32, state)
    phi = torch.ones((2, D), device=dev)
    tda.tda_precondition(tda.TDA_PC_FIT_ACCUM, 1, D, tda.TDA_F32, state, phi=phi, n=2, ld_phi=D)
    m = state[64:64 + 4 * D * D].view(torch.float32).view(D, D)
    m[3, 3] = -100.0
    q = torch.ones((2, D), device=dev)
    qh = torch.zeros((2, D), device=dev)
    tda.tda_precondition(tda.TDA_PC_FACTOR_APPLY, 1, D, tda.TDA_F32, state, n_total=2, lambda_abs=1e-3,
                         q=q, n_q=2, ld_q=D, qhat=qh, ld_qhat=D)
    with pytest.raises(tda.TdaError) as e:
        tda.tda_precondition_info(1, D, tda.TDA_F32, state)
    assert e.value.status == tda.TDA_ERR_NOT_SPD
    assert torch.isnan(qh).all()


def test_bounded_wait_times_out_and_context_survives(dev, orc):
    # a wait on a barrier nothing arrives on runs out after 50 ms; the error word reports it
    tda.tda_device_status()
    tda.tda_selftest_bounded_wait(50_000_000)
    with pytest.raises(tda.TdaError) as e:
        tda.tda_device_status()
    assert e.value.status == tda.TDA_ERR_TIMEOUT
    tda.tda_device_status()  # the word was cleared
    # the context is still usable: a projection afterwards matches the oracle
    A, B = make_factors(3, 40, 64, 64, "bf16", stream=12)
    L = tda.LayerDesc(64, 64, 40, 16, 16, seed=1, layer=1)
    got, _ = gpu_project(L, "bf16", to_dev(A, "bf16", dev), to_dev(B, "bf16", dev), 3, tda.TDA_ROUTE_FACTORED, dev)
    ref = orc.project(synth.to_f64(A, "bf16"), synth.to_f64(B, "bf16"), 16, 16, 1, 1)
    assert rel_fro(got, ref) <= TOL["bf16"]


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
@pytest.mark.parametrize("route", [tda.TDA_ROUTE_FACTORED, tda.TDA_ROUTE_MATERIALIZE, tda.TDA_ROUTE_GRAM,
                                   tda.TDA_ROUTE_AUTO])
def test_similarity_projected_routes_match_oracle(dev, orc, dtype, route):
    # projected-gradient inner products by the three routes (App. A.4), train side
    # streamed through a workspace that holds only a few examples at a time
    nq, nt, T, di, do, k = 3, 11, 37, 64, 48, 16
    Aq, Bq = make_factors(nq, T, di, do, dtype, stream=13, query=True)
    At, Bt = make_factors(nt, T, di, do, dtype, stream=13)
    L = tda.LayerDesc(di, do, T, k, k, seed=4, layer=2)
    base = tda.tda_workspace_size(tda.TDA_OP_SIMILARITY_PROJECTED, L, TD[dtype], nq, nt, route)
    wsb = base + 3 * (4 * k * k + 4 * T * 2 * k)  # room for a few more train examples per chunk
    ws = torch.empty(wsb, dtype=torch.uint8, device=dev)
    S = torch.full((nq, nt), 1.5, device=dev)
    tda.tda_similarity_projected(L, TD[dtype], to_dev(Aq, dtype, dev), to_dev(Bq, dtype, dev), nq,
                                 to_dev(At, dtype, dev), to_dev(Bt, dtype, dev), nt, S, nt, 2.0, route, ws, wsb)
    tda.tda_device_status()
    fq = orc.project(synth.to_f64(Aq, dtype), synth.to_f64(Bq, dtype), k, k, 4, 2)
    ft = orc.project(synth.to_f64(At, dtype), synth.to_f64(Bt, dtype), k, k, 4, 2)
    ref = orc.score(fq, ft) + 2.0 * 1.5
    assert rel_fro(S.cpu().numpy(), ref) <= TOL[dtype]


@pytest.mark.parametrize("nq,nt,D,beta", [(8, 64, 256, 0.0), (70, 300, 1024, 1.0), (64, 4096, 7168, 0.0),
                                          (3, 130, 100, 0.5), (200, 257, 64, 0.0),
                                          # more tiles than SMs with short K: the persistent kernel
                                          # (double-buffered accumulators), ragged edge tiles
                                          (300, 9000, 256, 0.0), (64, 20000, 512, 1.0), (129, 12001, 96, 0.5)])
def test_score_tensor_core_matches_oracle(dev, orc, nq, nt, D, beta):
    # fp32 scores on tcgen05 (3xTF32; cluster split-K, or one persistent CTA per SM walking
    # the tiles): within the fp32 tolerance
    rng = np.random.default_rng(nq + nt + D)
    Q = rng.standard_normal((nq, D)).astype(np.float32)
    P = (rng.standard_normal((nt, D)) * rng.uniform(0.1, 10.0, (nt, 1))).astype(np.float32)
    Qd, Pd = torch.from_numpy(Q).to(dev), torch.from_numpy(P).to(dev)
    assert tda.tda_score_engine(Qd, tda.TDA_F32, nq, D, Pd, nt, D, D) == 1
    S0 = rng.standard_normal((nq, nt)).astype(np.float32)
    S = torch.from_numpy(S0).to(dev)
    tda.tda_score(Qd, tda.TDA_F32, nq, D, Pd, nt, D, D, S, nt, beta=beta)
    tda.tda_device_status()
    ref = orc.score(Q, P) + beta * S0.astype(np.float64)
    assert rel_fro(S.cpu().numpy(), ref) <= 1e-5


@pytest.mark.gpu
@pytest.mark.parametrize("dtype", ["f32", "bf16"])
@pytest.mark.parametrize("op,route", [("proj", tda.TDA_ROUTE_FACTORED), ("proj", tda.TDA_ROUTE_MATERIALIZE),
                                      ("proj", tda.TDA_ROUTE_GRAM), ("exact", tda.TDA_ROUTE_MATERIALIZE),
                                      ("exact", tda.TDA_ROUTE_GRAM), ("proj", tda.TDA_ROUTE_AUTO)])
def test_norms_and_cosine_match_oracle(dev, orc, dtype, op, route):
    # per-example squared norms routed like Gram matrices (App. A.4), then cosine scores
    n, nq, T, di, do, k = 9, 3, 29, 64, 40, 16
    A, B = make_factors(n, T, di, do, dtype, stream=21)
    Aq, Bq = make_factors(nq, T, di, do, dtype, stream=21, query=True)
    L = tda.LayerDesc(di, do, T, k, k, seed=6, layer=1)
    opc = tda.TDA_OP_NORM_PROJECTED if op == "proj" else tda.TDA_OP_NORM_EXACT
    r = route if route != tda.TDA_ROUTE_AUTO else tda.tda_route(L, opc, n, 0, TD[dtype])[0]
    wsb = tda.tda_workspace_size(opc, L, TD[dtype], n, 0, r) * 3 + 256
    ws = torch.empty(max(wsb, 256), dtype=torch.uint8, device=dev)
    out = torch.full((n,), -1.0, device=dev)
    tda.tda_norms(opc, L, TD[dtype], to_dev(A, dtype, dev), to_dev(B, dtype, dev), n, out, route, ws, wsb)
    tda.tda_device_status()
    A64, B64 = synth.to_f64(A, dtype), synth.to_f64(B, dtype)
    if op == "proj":
        ref = (orc.project(A64, B64, k, k, 6, 1) ** 2).reshape(n, -1).sum(1)
    else:
        ref = orc.sq_norms(A64, B64, "materialized")
    tol = 1e-5 if dtype == "f32" else 2e-2
    np.testing.assert_allclose(out.cpu().numpy(), ref, rtol=tol)
    if op == "proj":
        # cosine of projected query/train features from device norms and scores
        nqd = torch.empty(nq, device=dev)
        tda.tda_norms(opc, L, TD[dtype], to_dev(Aq, dtype, dev), to_dev(Bq, dtype, dev), nq, nqd, route, ws, wsb)
        fq = orc.project(synth.to_f64(Aq, dtype), synth.to_f64(Bq, dtype), k, k, 6, 1)
        ft = orc.project(A64, B64, k, k, 6, 1)
        S0 = orc.score(fq, ft)
        S = torch.from_numpy(S0.astype(np.float32)).to(dev)
        tda.tda_cosine(S, nq, n, n, nqd, out)
        tda.tda_device_status()
        C = orc.cosine(S0, (fq ** 2).reshape(nq, -1).sum(1), ref)
        assert rel_fro(S.cpu().numpy(), C) <= (1e-5 if dtype == "f32" else 2e-2)
        assert np.abs(S.cpu().numpy()).max() <= 1 + 1e-5


@pytest.mark.gpu
def test_norms_edge_cases(dev, orc):
    # empty batch, T = 0 (zero gradients), a workspace that holds one example at a time
    L = tda.LayerDesc(32, 32, 0, 8, 8)
    out = torch.full((4,), 7.0, device=dev)
    z = torch.empty(16, device=dev)
    tda.tda_norms(tda.TDA_OP_NORM_EXACT, L, tda.TDA_F32, z, z, 4, out, tda.TDA_ROUTE_GRAM)
    tda.tda_norms(tda.TDA_OP_NORM_PROJECTED, L, tda.TDA_F32, z, z, 0, out, tda.TDA_ROUTE_FACTORED)
    tda.tda_device_status()
    assert (out.cpu() == 0).all()
    n, T, di, do = 5, 3, 24, 16
    A, B = make_factors(n, T, di, do, "f32", stream=22)
    L = tda.LayerDesc(di, do, T, 8, 8)
    wsb = tda.tda_workspace_size(tda.TDA_OP_NORM_EXACT, L, tda.TDA_F32, n, 0, tda.TDA_ROUTE_MATERIALIZE)
    ws = torch.empty(wsb, dtype=torch.uint8, device=dev)
    out = torch.empty(n, device=dev)
    tda.tda_norms(tda.TDA_OP_NORM_EXACT, L, tda.TDA_F32, to_dev(A, "f32", dev), to_dev(B, "f32", dev), n, out,
                  tda.TDA_ROUTE_MATERIALIZE, ws, wsb)
    tda.tda_device_status()
    np.testing.assert_allclose(out.cpu().numpy(), orc.sq_norms(A, B, "gram"), rtol=1e-5)


@pytest.mark.gpu
@pytest.mark.parametrize("nq,nt,T,di,do,beta", [
    (3, 37, 1, 64, 40, 0.0),      # 128 queries per tile row group of 1, 256 train per tile
    (5, 70, 8, 128, 64, 1.0),     # ragged query and train tiles
    (17, 33, 16, 64, 64, 0.0),    # three query tiles
    (3, 9, 32, 64, 128, 0.5),
    (4, 11, 64, 64, 64, 0.0),     # a query's rows span two epilogue warps
    (2, 5, 128, 136, 64, 1.0),    # ragged K chunk (136 = 2 x 64 + 8)
    (2, 3, 256, 64, 72, 0.0),     # one (query, train) pair per unit
    (2, 2, 512, 64, 64, 1.0),     # 4 x 2 tile pairs per unit
])
def test_gram_tensor_core_matches_oracle(dev, orc, nq, nt, T, di, do, beta):
    # route (c) of Eq. 4 on tcgen05: both token Grams as bf16 GEMMs, fp32 accumulation
    Aq, Bq = make_factors(nq, T, di, do, "bf16", stream=31, query=True)
    At, Bt = make_factors(nt, T, di, do, "bf16", stream=31)
    L = tda.LayerDesc(di, do, T, 1, 1)
    d = [to_dev(x, "bf16", dev) for x in (Aq, Bq, At, Bt)]
    assert tda.tda_similarity_gram_engine(L, tda.TDA_BF16, *d) == 1
    S0 = np.random.default_rng(T).standard_normal((nq, nt + 2)).astype(np.float32)
    S = torch.from_numpy(S0).to(dev)
    tda.tda_similarity_exact(L, tda.TDA_BF16, d[0], d[1], nq, d[2], d[3], nt, S, nt + 2, beta, tda.TDA_ROUTE_GRAM)
    tda.tda_device_status()
    ref = orc.similarity(*(synth.to_f64(x, "bf16") for x in (Aq, Bq, At, Bt))) + beta * S0[:, :nt]
    got = S.cpu().numpy()
    assert rel_fro(got[:, :nt], ref) <= 1e-5
    np.testing.assert_array_equal(got[:, nt:], S0[:, nt:])


# ------------------------------------------------------------------ K-FAC / EK-FAC
def _kfac_oracle(orc, A64, B64, k, seed, layer, kind, lam_abs, lam_rel, Q, phi64=None):
    Ca, Cg = orc.kfac_covariances(A64, B64, k, k, seed, layer)
    wa, Ua, _ = orc.sym_eig(Ca)
    wg, Ug, _ = orc.sym_eig(Cg)
    Lam = orc.kfac_eigenvalues(wa, wg) if kind == tda.TDA_KFAC else orc.ekfac_eigenvalues(phi64, Ua, Ug)
    lam = orc.kfac_damping(Lam, lam_abs, lam_rel)
    return Ca, Cg, wa, wg, orc.kfac_precondition(Ua, Ug, Lam, lam, Q)


@pytest.mark.gpu
@pytest.mark.parametrize("dtype,N,T,di,do,k,chunks", [("f32", 40, 13, 64, 48, 16, 3), ("bf16", 64, 32, 128, 64, 32, 2),
                                                     ("bf16", 9, 5, 64, 64, 64, 1), ("f32", 12, 7, 40, 24, 8, 2)])
@pytest.mark.parametrize("kind", [tda.TDA_KFAC, tda.TDA_EKFAC])
def test_kfac_ekfac_match_oracle(dev, orc, dtype, N, T, di, do, k, chunks, kind):
    # factor covariances streamed in chunks, Jacobi eigenbases, (EK-)FAC eigenvalues,
    # damping 0.1 x mean eigenvalue, preconditioned queries: the whole chain vs the oracle
    A, B = make_factors(N, T, di, do, dtype, stream=41, sigma_b=0.1, mask_p=0.02)
    L = tda.LayerDesc(di, do, T, k, k, seed=8, layer=5)
    Ad, Bd = to_dev(A, dtype, dev), to_dev(B, dtype, dev)
    st = torch.empty(tda.tda_kfac_state_bytes(k, k) // 8, dtype=torch.float64, device=dev)
    wsb = tda.tda_kfac_workspace_size(L, TD[dtype]) + 3 * 4 * T * 2 * k
    ws = torch.empty(wsb, dtype=torch.uint8, device=dev)
    tda.tda_kfac_reset(k, k, st)
    assert Ad.shape == (N, T, di)
    bounds = np.linspace(0, N, chunks + 1).astype(int)
    for e0, e1 in zip(bounds[:-1], bounds[1:]):
        tda.tda_kfac_accumulate_factors(L, TD[dtype], Ad[e0:], Bd[e0:], int(e1 - e0), st, ws, wsb)
    tda.tda_kfac_eigen(k, k, st)
    phi, _ = gpu_project(L, dtype, Ad, Bd, N, tda.TDA_ROUTE_FACTORED, dev)
    phid = torch.from_numpy(phi.astype(np.float32)).to(dev)
    if kind == tda.TDA_EKFAC:
        tda.tda_kfac_accumulate_eigenvalues(k, k, st, phid[: N // 2], N // 2, k * k, ws, wsb)
        tda.tda_kfac_accumulate_eigenvalues(k, k, st, phid[N // 2:], N - N // 2, k * k, ws, wsb)
    nq = 5
    Q = np.random.default_rng(k).standard_normal((nq, k * k)).astype(np.float32)
    Qd = torch.from_numpy(Q).to(dev)
    Qh = torch.full((nq, k * k + 3), float("nan"), device=dev)
    tda.tda_kfac_apply(kind, k, k, st, 0.0, 0.1, Qd, nq, k * k, Qh, k * k + 3)
    tda.tda_device_status()
    A64, B64 = synth.to_f64(A, dtype), synth.to_f64(B, dtype)
    phi64 = orc.project(A64, B64, k, k, 8, 5)
    Ca, Cg, wa, wg, ref = _kfac_oracle(orc, A64, B64, k, 8, 5, kind, 0.0, 0.1, Q, phi64)
    s = st.cpu().numpy()
    M = s[0]
    assert M == N * T
    assert s[2] >= 0 and s[3] >= 0  # both Jacobi runs converged
    np.testing.assert_allclose(s[8:8 + k * k].reshape(k, k) / M, Ca, rtol=2e-5, atol=1e-7 * np.abs(Ca).max())
    o = 8 + k * k
    np.testing.assert_allclose(s[o:o + k * k].reshape(k, k) / M, Cg, rtol=2e-5, atol=1e-7 * np.abs(Cg).max())
    o += k * k
    Ua = s[o:o + k * k].reshape(k, k)
    np.testing.assert_allclose(Ua.T @ Ua, np.eye(k), atol=1e-12)
    np.testing.assert_allclose(np.sort(s[o + k * k:o + k * k + k]), wa, rtol=1e-5, atol=1e-7 * wa.max())
    got = Qh.cpu().numpy()
    assert rel_fro(got[:, : k * k], ref) <= (1e-5 if dtype == "f32" else 1e-4)
    assert np.isnan(got[:, k * k:]).all()


@pytest.mark.gpu
@pytest.mark.parametrize("N,T,di,do,k", [(700, 256, 64, 128, 64), (300, 16, 128, 64, 32), (20, 300, 64, 72, 16)])
def test_project_kfac_fused_matches_oracle(dev, orc, N, T, di, do, k):
    # covariances accumulated inside the tensor-core projection (one pass over the factors)
    A, B = make_factors(N, T, di, do, "bf16", stream=43, sigma_b=0.05, mask_p=0.01)
    L = tda.LayerDesc(di, do, T, k, k, seed=2, layer=1)
    Ad, Bd = to_dev(A, "bf16", dev), to_dev(B, "bf16", dev)
    st = torch.empty(tda.tda_kfac_state_bytes(k, k) // 8, dtype=torch.float64, device=dev)
    wsb = tda.tda_kfac_workspace_size(L, tda.TDA_BF16)
    ws = torch.empty(wsb, dtype=torch.uint8, device=dev)
    phi = torch.full((N, k * k), float("nan"), device=dev)
    tda.tda_kfac_reset(k, k, st)
    tda.tda_project_kfac(L, tda.TDA_BF16, Ad, Bd, N, phi, k * k, st, ws, wsb)
    tda.tda_device_status()
    A64, B64 = synth.to_f64(A, "bf16"), synth.to_f64(B, "bf16")
    ref_phi = orc.project(A64, B64, k, k, 2, 1)
    assert rel_fro(phi.cpu().numpy().reshape(ref_phi.shape), ref_phi) <= 1e-5
    Ca, Cg = orc.kfac_covariances(A64, B64, k, k, 2, 1)
    s = st.cpu().numpy()
    assert s[0] == N * T
    assert rel_fro(s[8:8 + k * k].reshape(k, k) / s[0], Ca) <= 1e-5
    assert rel_fro(s[8 + k * k:8 + 2 * k * k].reshape(k, k) / s[0], Cg) <= 1e-5


@pytest.mark.gpu
@pytest.mark.parametrize("kind", [tda.TDA_KFAC, tda.TDA_EKFAC])
def test_kfac_batched_layers_match_oracle(dev, orc, kind):
    # three linears of one block in one state buffer: fused projection per linear, then
    # eigenbases, EK-FAC sums and the preconditioner for all linears in one launch each
    N, T, k, nq = 160, 64, 32, 6
    shapes = [(128, 128), (128, 256), (256, 128)]
    D = k * k
    per = tda.tda_kfac_state_bytes(k, k)
    st = torch.empty(len(shapes) * per // 8, dtype=torch.float64, device=dev)
    Ls = [tda.LayerDesc(di, do, T, k, k, seed=3, layer=i) for i, (di, do) in enumerate(shapes)]
    wsb = max(tda.tda_kfac_workspace_size(L, tda.TDA_BF16) for L in Ls)
    ws = torch.empty(wsb, dtype=torch.uint8, device=dev)
    Phi = torch.empty((N, len(shapes) * D), device=dev)
    tda.tda_kfac_reset(k, k, st, n_layers=len(shapes))
    facts = []
    for i, (L, (di, do)) in enumerate(zip(Ls, shapes)):
        A, B = make_factors(N, T, di, do, "bf16", stream=50 + i, sigma_b=0.05)
        facts.append((synth.to_f64(A, "bf16"), synth.to_f64(B, "bf16")))
        tda.tda_project_kfac(L, tda.TDA_BF16, to_dev(A, "bf16", dev), to_dev(B, "bf16", dev), N, Phi[:, i * D:],
                             len(shapes) * D, st[i * per // 8:], ws, wsb)
    tda.tda_kfac_eigen(k, k, st, n_layers=len(shapes))
    if kind == tda.TDA_EKFAC:
        tda.tda_kfac_accumulate_eigenvalues(k, k, st, Phi, N, len(shapes) * D, ws, wsb, n_layers=len(shapes))
    Q = np.random.default_rng(1).standard_normal((nq, len(shapes) * D)).astype(np.float32)
    Qh = torch.empty((nq, len(shapes) * D), device=dev)
    tda.tda_kfac_apply(kind, k, k, st, 0.0, 0.1, torch.from_numpy(Q).to(dev), nq, len(shapes) * D, Qh,
                       len(shapes) * D, n_layers=len(shapes))
    tda.tda_device_status()
    got = Qh.cpu().numpy()
    for i, (A64, B64) in enumerate(facts):
        phi64 = orc.project(A64, B64, k, k, 3, i)
        ref = _kfac_oracle(orc, A64, B64, k, 3, i, kind, 0.0, 0.1, Q[:, i * D:(i + 1) * D], phi64)[-1]
        assert rel_fro(got[:, i * D:(i + 1) * D], ref) <= 1e-4, i


# ------------------------------------------------------------------ token scores / masks
@pytest.mark.gpu
@pytest.mark.parametrize("dtype,N,T,di,do,k,kind", [("f32", 5, 70, 64, 48, 16, 0), ("bf16", 4, 130, 128, 64, 32, 0),
                                                    ("f32", 3, 9, 24, 16, 24, 1)])
def test_token_scores_match_oracle(dev, orc, dtype, N, T, di, do, k, kind):
    # s_t = g~_t^T R a~_t per token; beta = 1 accumulates a second layer's share
    ko = do if kind == 1 else k
    ki = di if kind == 1 else k
    A, B = make_factors(N, T, di, do, dtype, stream=61, sigma_b=0.1, mask_p=0.05)
    L = tda.LayerDesc(di, do, T, ki, ko, seed=7, layer=4, kind=kind)
    nq = 3
    R = np.random.default_rng(T).standard_normal((nq, ko, ki)).astype(np.float32)
    Rd = torch.from_numpy(R.reshape(nq, -1)).to(dev)
    out0 = np.random.default_rng(1).standard_normal((nq, N * T + 5)).astype(np.float32)
    out = torch.from_numpy(out0).to(dev)
    wsb = tda.tda_token_scores_workspace_size(L) * 2
    ws = torch.empty(wsb, dtype=torch.uint8, device=dev)
    tda.tda_token_scores(L, TD[dtype], to_dev(A, dtype, dev), to_dev(B, dtype, dev), N, Rd, nq, ki * ko, out,
                         N * T + 5, 1.0, ws, wsb)
    tda.tda_device_status()
    A64, B64 = synth.to_f64(A, dtype), synth.to_f64(B, dtype)
    ref = orc.token_scores(A64, B64, R, ki, ko, 7, 4, kind)
    got = out.cpu().numpy()
    assert rel_fro(got[:, : N * T].reshape(nq, N, T) - out0[:, : N * T].reshape(nq, N, T), ref) <= 1e-5
    np.testing.assert_array_equal(got[:, N * T:], out0[:, N * T:])
    # the decomposition sums to the sequence-level score
    phi = orc.project(A64, B64, ki, ko, 7, 4, kind)
    np.testing.assert_allclose(ref.sum(2), orc.score(R, phi), rtol=1e-10)


@pytest.mark.gpu
@pytest.mark.parametrize("dtype,N,T,di,do,ki,ko,nq", [("bf16", 64, 512, 128, 64, 32, 32, 9),
                                                      ("f32", 7, 45, 96, 80, 32, 16, 11),
                                                      ("bf16", 5, 77, 64, 128, 32, 64, 5)])
def test_token_scores_tensor_core_shapes(dev, orc, dtype, N, T, di, do, ki, ko, nq):
    # k_in = 32 runs on the tensor cores: several token tiles per CTA (first case), several query
    # stages of 256 (q, r) rows, k_out = 16 / 32 / 64, ragged token and query tails; beta = 0.5
    A, B = make_factors(N, T, di, do, dtype, stream=63, sigma_b=0.1, mask_p=0.05)
    L = tda.LayerDesc(di, do, T, ki, ko, seed=11, layer=2)
    R = np.random.default_rng(N + T).standard_normal((nq, ko, ki)).astype(np.float32)
    Rd = torch.from_numpy(R.reshape(nq, -1)).to(dev)
    out0 = np.random.default_rng(2).standard_normal((nq, N * T + 3)).astype(np.float32)
    out = torch.from_numpy(out0).to(dev)
    wsb = tda.tda_token_scores_workspace_size(L) * N + (1 << 20)
    ws = torch.empty(wsb, dtype=torch.uint8, device=dev)
    tda.tda_token_scores(L, TD[dtype], to_dev(A, dtype, dev), to_dev(B, dtype, dev), N, Rd, nq, ki * ko, out,
                         N * T + 3, 0.5, ws, wsb)
    tda.tda_device_status()
    ref = orc.token_scores(synth.to_f64(A, dtype), synth.to_f64(B, dtype), R, ki, ko, 11, 2, 0)
    got = out.cpu().numpy()
    assert rel_fro(got[:, : N * T].reshape(nq, N, T) - 0.5 * out0[:, : N * T].reshape(nq, N, T), ref) <= 1e-5
    np.testing.assert_array_equal(got[:, N * T:], out0[:, N * T:])


@pytest.mark.gpu
@pytest.mark.parametrize("dtype,N,T,di,do,nc", [("bf16", 6, 37, 256, 128, 20000), ("f32", 3, 100, 64, 80, 700)])
def test_mask_gather_matches_oracle(dev, orc, dtype, N, T, di, do, nc):
    # entries of DW at random coordinates, gathered from the factors; invalid coordinates -> NaN
    A, B = make_factors(N, T, di, do, dtype, stream=62, sigma_b=0.1)
    rng = np.random.default_rng(nc)
    rows = rng.integers(0, do, nc).astype(np.int32)
    cols = rng.integers(0, di, nc).astype(np.int32)
    rows[5], cols[7] = do, -1
    L = tda.LayerDesc(di, do, T, 1, 1)
    out = torch.full((N, nc + 2), 3.0, device=dev)
    tda.tda_mask_gather(L, TD[dtype], to_dev(A, dtype, dev), to_dev(B, dtype, dev), N,
                        torch.from_numpy(rows).to(dev), torch.from_numpy(cols).to(dev), nc, out, nc + 2)
    tda.tda_device_status()
    got = out.cpu().numpy()
    ok = np.ones(nc, bool)
    ok[[5, 7]] = False
    ref = orc.mask_gather(synth.to_f64(A, dtype), synth.to_f64(B, dtype), np.where(ok, rows, 0), np.where(ok, cols, 0))
    assert rel_fro(got[:, :nc][:, ok], ref[:, ok]) <= 1e-5
    assert np.isnan(got[:, 5]).all() and np.isnan(got[:, 7]).all()
    assert (got[:, nc:] == 3.0).all()


@pytest.mark.gpu
@pytest.mark.parametrize("kind", [tda.TDA_KFAC, tda.TDA_EKFAC])
def test_kfac_without_curvature_is_damping_only(dev, kind):
    # degenerate case: no training tokens seen (M = 0): C_a = C_g = 0, every eigenvalue is 0,
    # so the preconditioner is lambda_abs^-1 I and Qhat = Q / lambda_abs
    k = 16
    st = torch.empty(tda.tda_kfac_state_bytes(k, k) // 8, dtype=torch.float64, device=dev)
    tda.tda_kfac_reset(k, k, st)
    tda.tda_kfac_eigen(k, k, st)
    Q = torch.randn(3, k * k, device=dev)
    Qh = torch.empty_like(Q)
    tda.tda_kfac_apply(kind, k, k, st, 0.5, 0.1, Q, 3, k * k, Qh, k * k)
    tda.tda_device_status()
    s = st.cpu().numpy()
    assert s[2] == 0 and s[3] == 0  # Jacobi: already diagonal, zero sweeps
    torch.testing.assert_close(Qh, Q / 0.5, rtol=1e-6, atol=1e-7)


@pytest.mark.gpu
@pytest.mark.parametrize("N,T,di,do,k", [(3, 70, 264, 136, 16), (2, 37, 512, 200, 32), (5, 130, 256, 128, 8)])
def test_materialize_route_tensor_core_matches_oracle(dev, orc, N, T, di, do, k):
    # route (b) for bf16: DW built by the tensor-core kernel (ragged rows, columns and token chunks),
    # then projected; also the exact norms and similarities that materialise DW
    A, B = make_factors(N, T, di, do, "bf16", stream=71, sigma_b=0.1, mask_p=0.02)
    L = tda.LayerDesc(di, do, T, k, k, seed=9, layer=6)
    Ad, Bd = to_dev(A, "bf16", dev), to_dev(B, "bf16", dev)
    got, _ = gpu_project(L, "bf16", Ad, Bd, N, tda.TDA_ROUTE_MATERIALIZE, dev)
    A64, B64 = synth.to_f64(A, "bf16"), synth.to_f64(B, "bf16")
    assert rel_fro(got, orc.project(A64, B64, k, k, 9, 6)) <= 1e-5
    wsb = tda.tda_workspace_size(tda.TDA_OP_NORM_EXACT, L, tda.TDA_BF16, N, 0, tda.TDA_ROUTE_MATERIALIZE) * 2
    ws = torch.empty(wsb, dtype=torch.uint8, device=dev)
    nrm = torch.empty(N, device=dev)
    tda.tda_norms(tda.TDA_OP_NORM_EXACT, L, tda.TDA_BF16, Ad, Bd, N, nrm, tda.TDA_ROUTE_MATERIALIZE, ws, wsb)
    tda.tda_device_status()
    np.testing.assert_allclose(nrm.cpu().numpy(), orc.sq_norms(A64, B64, "materialized"), rtol=1e-5)
