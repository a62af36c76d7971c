"""Parity at the workloads' full sizes, on sampled outputs the oracle computes
one by one, and stage by stage from the GPU's own features.

* Llama-1B block (the benchmark's workload and launch configuration): 4096 train
  and 64 query examples resident, the whole pass of BlockPipeline; sampled
  feature rows and GradDot scores against the oracle; then, from the GPU's
  downloaded features, the oracle's fp64 damping, preconditioned queries and
  preconditioned score matrix, compared with the GPU's S; top-k selection
  bit-exact on the GPU's S and consistent with the oracle's S wherever the
  score gaps exceed the measured score error.
* Llama-3-8B layer shapes (k = 64, T = 1024): one streamed chunk of 256 train
  examples through the 7 linears of a layer, with 16 and with all 256 queries.
* Large-model block (d_model 12288, ffn 49152, GQA k/v 12288 -> 1536; k = 128,
  T = 2048, Student-t activations): 7 x 16384 features per example, the
  D = 16384 Fisher fit, factorisation and query solves, the preconditioned
  score and the top-100; the factors are also streamed from pinned host memory.
* The 8192 x 8192 linear of the route sweep: exact similarity by both routes at
  T = 8 ... 512, the projection by both routes at T = 8 and 2048.
Tolerances: relative Frobenius error 2e-2 for score matrices and features from bf16 factors
(fp32 accumulation).
"""
import math
import os

import numpy as np
import pytest
import torch

import paper_2609_38767_gb300 as tda
from paper_2609_38767_gb300 import build as tbuild
from paper_2609_38767_gb300 import synth
from paper_2609_38767_gb300.block import BlockPipeline

pytestmark = pytest.mark.gpu
TOL = 2e-2


@pytest.fixture(scope="module")
def dev():
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    tbuild.build()
    tda.load()
    return torch.device("cuda:0")


def rel_fro(x, ref):
    x, ref = np.asarray(x, np.float64), np.asarray(ref, np.float64)
    return float(np.linalg.norm(x - ref) / np.linalg.norm(ref))


def fill(n, T, d, seed, stream, sigma, dist, mask_p, mask_stream, dev):
    x = torch.empty(n * T * d, dtype=torch.bfloat16, device=dev)
    synth.fill_device(x, seed, stream, n, T, d, sigma, dist, 0, mask_p, mask_stream=mask_stream)
    return x


def oracle_example(orc, e, role, li, T, di, do, k, sig_b, dist_a, mask_p, layer):
    off, ms = (synth.QUERY_STREAM_OFFSET, 1000) if role == "query" else (0, 0)
    A = synth.factors(synth.SEED_A, li + off, 1, T, di, 1.0, dist_a, e, "bf16", mask_p, mask_stream=ms)
    B = synth.factors(synth.SEED_B, li + off, 1, T, do, sig_b, 0, e, "bf16", mask_p, mask_stream=ms)
    return orc.project(synth.to_f64(A, "bf16"), synth.to_f64(B, "bf16"), k, k, 0, layer)[0].reshape(-1)


def run_block(dev, linears, T, k, N, Nq, sig_b, dist_a, mask_p, topk):
    At, Bt, Aq, Bq = [], [], [], []
    for li, (di, do) in enumerate(linears):
        At.append(fill(N, T, di, synth.SEED_A, li, 1.0, dist_a, mask_p, 0, dev))
        Bt.append(fill(N, T, do, synth.SEED_B, li, sig_b, 0, mask_p, 0, dev))
        Aq.append(fill(Nq, T, di, synth.SEED_A, li + synth.QUERY_STREAM_OFFSET, 1.0, dist_a, mask_p, 1000, dev))
        Bq.append(fill(Nq, T, do, synth.SEED_B, li + synth.QUERY_STREAM_OFFSET, sig_b, 0, mask_p, 1000, dev))
    pipe = BlockPipeline(linears, T, k, N, Nq, topk=topk, precondition=True, lambda_rel=1e-2, device=dev)
    for li, L in enumerate(pipe.layers):
        assert tda.tda_project_engine(L, tda.TDA_BF16, At[li], Bt[li]) == 1
    pipe.run(lambda li, L, r, phi, ld: tda.tda_project(L, tda.TDA_BF16, At[li], Bt[li], N, phi, ld, r),
             lambda li, L, r, phi, ld: tda.tda_project(L, tda.TDA_BF16, Aq[li], Bq[li], Nq, phi, ld, r))
    S_plain = torch.empty((Nq, N), device=dev)  # GradDot (unpreconditioned) on the same features
    tda.tda_score(pipe.Q, tda.TDA_F32, Nq, pipe.DT, pipe.Phi, N, pipe.DT, pipe.DT, S_plain, N)
    info = tda.tda_precondition_info(pipe.nl, pipe.D, tda.TDA_F32, pipe.state)
    tda.tda_device_status()
    del At, Bt, Aq, Bq
    return pipe, S_plain, info


def topk_against_reference_scores(idx, S_gpu, S_ref, k):
    """Top-k test against the oracle's fp64 scores: at every rank whose oracle score is
    more than twice the row's measured score error away from both neighbours, the GPU's
    index must be the oracle's; returns the number of ranks where the two differ (swaps
    among scores closer than the error)."""
    oi, ov = _orc_topk(S_ref, k + 1)
    swaps = 0
    for q in range(S_ref.shape[0]):
        err = float(np.abs(S_gpu[q].astype(np.float64) - S_ref[q]).max())
        for r in range(k):
            gap = ov[q, r] - ov[q, r + 1]
            if r > 0:
                gap = min(gap, ov[q, r - 1] - ov[q, r])
            if gap > 2 * err:
                assert idx[q, r] == oi[q, r], (q, r, err, gap)
            elif idx[q, r] != oi[q, r]:
                swaps += 1
    return swaps


_ORC = None


def _orc_topk(S, k):
    return _ORC.topk(S, k)


def stagewise(orc, pipe, info, lam_rel=1e-2):
    """F, lambda, Qhat and S recomputed in fp64 by the oracle from the GPU's features, per
    linear (D x D Cholesky when N >= D, its Woodbury form otherwise); S compared with the
    GPU's preconditioned score matrix, the top-k with the oracle's scores."""
    global _ORC
    _ORC = orc
    orc.set_threads(os.cpu_count() or 1)
    D, N = pipe.D, pipe.N
    Phi64 = pipe.Phi.cpu().numpy().astype(np.float64)
    Q64 = pipe.Q.cpu().numpy().astype(np.float64)
    Qh = pipe.Qh.cpu().numpy().astype(np.float64)
    Qh_ref = np.empty_like(Q64)
    for li in range(pipe.nl):
        sl = slice(li * D, (li + 1) * D)
        P = np.ascontiguousarray(Phi64[:, sl])
        lam = orc.damping_features(P, 0.0, lam_rel)
        assert abs(info[4 * li] - lam) <= 1e-4 * lam, li
        Ql = np.ascontiguousarray(Q64[:, sl])
        Qh_ref[:, sl] = orc.precondition(orc.fisher(P), lam, Ql) if N >= D else orc.precondition_lowrank(P, lam, Ql)
        assert rel_fro(Qh[:, sl], Qh_ref[:, sl]) <= TOL, ("qhat", li)
    S_ref = orc.score(Qh_ref, Phi64)
    S = pipe.S.cpu().numpy()
    err = rel_fro(S, S_ref)
    assert err <= TOL, err
    swaps = topk_against_reference_scores(pipe.idx.cpu().numpy(), S, S_ref, pipe.topk)
    print(f"preconditioned S: rel. Frobenius error {err:.2e}; top-{pipe.topk} swaps among near-ties: {swaps}")
    return err, swaps


def check_block(orc, pipe, S_plain, info, linears, T, k, sig_b, dist_a, mask_p, train_s, query_s, rng):
    D, N, Nq = k * k, pipe.N, pipe.Nq
    phi = {e: pipe.Phi[e].cpu().numpy() for e in train_s}
    qf = {e: pipe.Q[e].cpu().numpy() for e in query_s}
    ophi = {e: np.concatenate([oracle_example(orc, e, "train", li, T, di, do, k, sig_b, dist_a, mask_p, li)
                               for li, (di, do) in enumerate(linears)]) for e in train_s}
    oq = {e: np.concatenate([oracle_example(orc, e, "query", li, T, di, do, k, sig_b, dist_a, mask_p, li)
                             for li, (di, do) in enumerate(linears)]) for e in query_s}
    for e in train_s:
        assert rel_fro(phi[e], ophi[e]) <= TOL, ("train", e)
        for li in range(len(linears)):
            assert rel_fro(phi[e][li * D:(li + 1) * D], ophi[e][li * D:(li + 1) * D]) <= TOL
    for e in query_s:
        assert rel_fro(qf[e], oq[e]) <= TOL, ("query", e)
    # GradDot scores of the sampled pairs, oracle features on both sides
    Sp = S_plain.cpu().numpy()
    got = np.array([[Sp[q, i] for i in train_s] for q in query_s])
    ref = np.array([[float(oq[q] @ ophi[i]) for i in train_s] for q in query_s])
    assert rel_fro(got, ref) <= TOL
    # top-k: selection on the GPU's own score matrix is bit-exact
    S = pipe.S.cpu().numpy()
    oi, ov = orc.topk(S.astype(np.float64), pipe.topk)
    np.testing.assert_array_equal(pipe.idx.cpu().numpy(), oi)
    np.testing.assert_array_equal(pipe.val.cpu().numpy(), ov.astype(np.float32))
    # the solve: (F + lambda I) qhat = q for every linear, F from the features it was fitted on
    Phi64 = pipe.Phi.cpu().numpy().astype(np.float64)
    Qh = pipe.Qh.cpu().numpy().astype(np.float64)
    Q = pipe.Q.cpu().numpy().astype(np.float64)
    for li in range(len(linears)):
        P = Phi64[:, li * D:(li + 1) * D]
        tr = float((P * P).sum()) / N
        lam = 1e-2 * tr / D
        assert abs(info[4 * li] - lam) <= 1e-4 * lam
        X = Qh[:, li * D:(li + 1) * D]
        R = (X @ P.T) @ P / N + lam * X - Q[:, li * D:(li + 1) * D]
        assert np.linalg.norm(R) <= 1e-3 * np.linalg.norm(Q[:, li * D:(li + 1) * D]), li
    # stage by stage against the oracle: F, lambda, Qhat and the preconditioned S
    stagewise(orc, pipe, info)
    return got, ref


LLAMA1B = [(2048, 2048)] * 4 + [(2048, 8192)] * 2 + [(8192, 2048)]
LLAMA8B = [(4096, 4096), (4096, 1024), (4096, 1024), (4096, 4096), (4096, 14336), (4096, 14336), (14336, 4096)]


def test_llama1b_block_full_size(dev, orc):
    # 4096 train / 64 query, T = 512, k = 32, B ~ N(0, 1e-3), 1% masked tokens
    sb = math.sqrt(1e-3)
    pipe, S_plain, info = run_block(dev, LLAMA1B, 512, 32, 4096, 64, sb, 0, 0.01, 100)
    rng = np.random.default_rng(0)
    train_s = [0, int(rng.integers(1, 4095)), 4095]
    check_block(orc, pipe, S_plain, info, LLAMA1B, 512, 32, sb, 0, 0.01, train_s, [0, 63], rng)


@pytest.mark.parametrize("Nq", [16, 256])
def test_llama8b_layer_chunk_full_shapes(dev, orc, Nq):
    # one streamed chunk of 256 train examples, T = 1024, k = 64; 16 queries, or all 256 of the
    # workload (the blocked D = 4096 solve with a full query tile count)
    pipe, S_plain, info = run_block(dev, LLAMA8B, 1024, 64, 256, Nq, 0.1, 0, 0.0, 100)
    check_block(orc, pipe, S_plain, info, LLAMA8B, 1024, 64, 0.1, 0, 0.0, [0, 255], [7], np.random.default_rng(1))


LARGE = [(12288, 12288), (12288, 1536), (12288, 1536), (12288, 12288), (12288, 49152), (12288, 49152),
         (49152, 12288)]


def test_large_model_block_preconditioned_top100(dev, orc):
    # the large-model block at full width: T = 2048, k = 128 (D = 16384 per linear), A ~ Student-t(4),
    # B ~ N(0, 1e-4); 2048 train and 32 query examples (the full 16384 x 512 workload's factors do not
    # fit the device), factors generated on the device one 256-example chunk at a time;
    # lambda = 1e-2 x mean eigenvalue; preconditioned 32 x 2048 score and top-100 per query.
    # With fewer train examples than features F has rank N: the fp32 rounding of Qhat's large
    # component along F's null space (about q / lambda) reaches S with a weight that grows like
    # (D/N)^1.5 / lambda_rel; at N = 256 it alone is ~5% of S, at N = 2048 ~0.2%.
    T, k, N, Nq, sb, CH = 2048, 128, 2048, 32, 0.01, 256
    dist = synth.DIST_STUDENT_T4
    pipe = BlockPipeline(LARGE, T, k, N, Nq, topk=100, precondition=True, lambda_rel=1e-2, device=dev)

    def proj(role):
        n_all, off, ms = (N, 0, 0) if role == "train" else (Nq, synth.QUERY_STREAM_OFFSET, 1000)

        def f(li, L, route, phi, ld):
            di, do = LARGE[li]
            for c0 in range(0, n_all, CH):
                n = min(CH, n_all - c0)
                A = torch.empty(n * T * di, dtype=torch.bfloat16, device=dev)
                B = torch.empty(n * T * do, dtype=torch.bfloat16, device=dev)
                synth.fill_device(A, synth.SEED_A, li + off, n, T, di, 1.0, dist, e0=c0, mask_stream=ms)
                synth.fill_device(B, synth.SEED_B, li + off, n, T, do, sb, 0, e0=c0, mask_stream=ms)
                assert tda.tda_project_engine(L, tda.TDA_BF16, A, B) == 1
                tda.tda_project(L, tda.TDA_BF16, A, B, n, phi[c0:], ld, route)
                torch.cuda.synchronize()
                del A, B
        return f

    pipe.run(proj("train"), proj("query"))
    info = tda.tda_precondition_info(pipe.nl, pipe.D, tda.TDA_F32, pipe.state)
    tda.tda_device_status()
    # sampled features against the oracle (the narrow k/v linear, train examples in two chunks, a query)
    D = k * k
    for role, e in (("train", 3), ("train", 1500), ("query", 5)):
        ref = oracle_example(orc, e, role, 1, T, 12288, 1536, k, sb, dist, 0.0, 1)
        got = (pipe.Phi if role == "train" else pipe.Q)[e, D:2 * D].cpu().numpy()
        assert rel_fro(got, ref) <= TOL, (role, e)
    # top-100 selection bit-exact on the GPU's own scores
    S = pipe.S.cpu().numpy()
    oi, ov = orc.topk(S.astype(np.float64), 100)
    np.testing.assert_array_equal(pipe.idx.cpu().numpy(), oi)
    np.testing.assert_array_equal(pipe.val.cpu().numpy(), ov.astype(np.float32))
    stagewise(orc, pipe, info)


@pytest.mark.parametrize("li,di,do,pws", [(1, 12288, 1536, False), (4, 12288, 49152, False),
                                          (1, 12288, 1536, True)])
def test_large_model_layer_from_pinned_host(dev, orc, li, di, do, pws):
    # T = 2048, k = 128, A ~ Student-t(4), B ~ N(0, 1e-4); factors in pinned host memory.
    # pws: room for the projection's own workspace beside the staging halves (sign tables,
    # balanced token-tile ranges: 2 examples' 32 tiles over 32 SMs)
    T, k, n, sb = 2048, 128, 2, 0.01
    A = synth.factors(synth.SEED_A, li, n, T, di, 1.0, synth.DIST_STUDENT_T4, 0, "bf16")
    B = synth.factors(synth.SEED_B, li, n, T, do, sb, 0, 0, "bf16")
    Ah = torch.from_numpy(A.view(np.int16)).view(torch.bfloat16).pin_memory()
    Bh = torch.from_numpy(B.view(np.int16)).view(torch.bfloat16).pin_memory()
    L = tda.LayerDesc(di, do, T, k, k, seed=0, layer=li)
    wsb = 2 * tda.tda_project_host_ws_min(L, tda.TDA_BF16)
    if pws:
        p = tda.tda_workspace_size(tda.TDA_OP_PROJECT, L, tda.TDA_BF16, n, 0, tda.TDA_ROUTE_FACTORED)
        wsb += 2 * ((p + 255) // 256 * 256)
    ws = torch.empty(wsb, dtype=torch.uint8, device=dev)
    phi = torch.empty((n, k * k), device=dev)
    tda.tda_project_host(L, tda.TDA_BF16, Ah, Bh, n, phi, k * k, ws, wsb)
    tda.tda_device_status()
    ref = orc.project(synth.to_f64(A, "bf16"), synth.to_f64(B, "bf16"), k, k, 0, li)
    got = phi.cpu().numpy().reshape(n, k, k)
    for e in range(n):
        assert rel_fro(got[e], ref[e]) <= TOL


def test_llama8b_gate_from_pinned_host_small_pieces(dev, orc):
    # the Llama-3-8B stack's e2e leg: 4-example pieces of the gate linear (4096 -> 14336,
    # T = 1024, k = 64) from pinned host memory, with the projection's workspace beside the
    # staging halves (balanced token-tile ranges: 32 tiles over 32 SMs, no example split)
    T, k, n, li = 1024, 64, 4, 4
    di, do = 4096, 14336
    A = synth.factors(synth.SEED_A, li, n, T, di, 1.0, 0, 0, "bf16")
    B = synth.factors(synth.SEED_B, li, n, T, do, math.sqrt(1e-3), 0, 0, "bf16")
    Ah = torch.from_numpy(A.view(np.int16)).view(torch.bfloat16).pin_memory()
    Bh = torch.from_numpy(B.view(np.int16)).view(torch.bfloat16).pin_memory()
    L = tda.LayerDesc(di, do, T, k, k, seed=0, layer=li)
    p = tda.tda_workspace_size(tda.TDA_OP_PROJECT, L, tda.TDA_BF16, n, 0, tda.TDA_ROUTE_FACTORED)
    wsb = n * tda.tda_project_host_ws_min(L, tda.TDA_BF16) + 2 * ((p + 255) // 256 * 256)
    ws = torch.empty(wsb, dtype=torch.uint8, device=dev)
    phi = torch.empty((n, k * k), device=dev)
    for _ in range(2):  # the second call reuses the staging halves and the projection workspaces
        tda.tda_project_host(L, tda.TDA_BF16, Ah, Bh, n, phi, k * k, ws, wsb)
    tda.tda_device_status()
    ref = orc.project(synth.to_f64(A, "bf16"), synth.to_f64(B, "bf16"), k, k, 0, li)
    got = phi.cpu().numpy().reshape(n, k, k)
    for e in range(n):
        assert rel_fro(got[e], ref[e]) <= TOL


def test_topk_at_large_model_query_shape(dev, orc):
    # 512 queries x 16384 train, top-100, descending with ties to the lower index
    rng = np.random.default_rng(2)
    S = (rng.standard_normal((512, 16384)) * 32).round().astype(np.float32)  # many exact ties
    Sd = torch.from_numpy(S).to(dev)
    idx = torch.empty((512, 100), dtype=torch.int32, device=dev)
    val = torch.empty((512, 100), device=dev)
    tda.tda_topk(Sd, 512, 16384, 16384, 100, idx, val)
    oi, ov = orc.topk(S.astype(np.float64), 100)
    np.testing.assert_array_equal(idx.cpu().numpy(), oi)
    np.testing.assert_array_equal(val.cpu().numpy(), ov.astype(np.float32))


@pytest.mark.parametrize("T", [8, 32, 128, 512])
def test_route_sweep_linear_exact_similarity(dev, orc, T):
    # 8192 x 8192 linear, A, B ~ N(0, 1): Gram route and materialise route vs the oracle
    d, nq, nt = 8192, 2, 2
    Aq = synth.factors(synth.SEED_A, 1000, nq, T, d, 1.0, dtype="bf16")
    Bq = synth.factors(synth.SEED_B, 1000, nq, T, d, 1.0, dtype="bf16")
    At = synth.factors(synth.SEED_A, 0, nt, T, d, 1.0, dtype="bf16")
    Bt = synth.factors(synth.SEED_B, 0, nt, T, d, 1.0, dtype="bf16")
    to = lambda x: torch.from_numpy(x.view(np.int16)).view(torch.bfloat16).to(dev)
    L = tda.LayerDesc(d, d, T, 1, 1)
    ref = orc.similarity(synth.to_f64(Aq, "bf16"), synth.to_f64(Bq, "bf16"), synth.to_f64(At, "bf16"),
                         synth.to_f64(Bt, "bf16"))
    for route in (tda.TDA_ROUTE_GRAM, tda.TDA_ROUTE_MATERIALIZE):
        wsb = max(tda.tda_workspace_size(tda.TDA_OP_SIMILARITY_EXACT, L, tda.TDA_BF16, nq, nt, route), 1)
        ws = torch.empty(wsb, dtype=torch.uint8, device=dev)
        S = torch.empty((nq, nt), device=dev)
        tda.tda_similarity_exact(L, tda.TDA_BF16, to(Aq), to(Bq), nq, to(At), to(Bt), nt, S, nt, 0.0, route, ws, wsb)
        tda.tda_device_status()
        assert rel_fro(S.cpu().numpy(), ref) <= TOL, route


@pytest.mark.parametrize("T", [8, 2048])
def test_route_sweep_linear_projection_both_routes(dev, orc, T):
    # the 8192 x 8192 linear of the route sweep at a short and a long T, k = 64, A, B ~ N(0, 1): the
    # factored tensor-core projection and the materialise route against the oracle (at T = 8192 the
    # oracle's loops take minutes per example)
    d, n, k = 8192, 2, 64
    A = synth.factors(synth.SEED_A, 0, n, T, d, 1.0, dtype="bf16")
    B = synth.factors(synth.SEED_B, 0, n, T, d, 1.0, dtype="bf16")
    to = lambda x: torch.from_numpy(x.view(np.int16)).view(torch.bfloat16).to(dev)
    L = tda.LayerDesc(d, d, T, k, k, seed=0, layer=0)
    orc.set_threads(os.cpu_count() or 1)
    ref = orc.project(synth.to_f64(A, "bf16"), synth.to_f64(B, "bf16"), k, k, 0, 0).reshape(n, k * k)
    Ad, Bd = to(A), to(B)
    assert tda.tda_project_engine(L, tda.TDA_BF16, Ad, Bd) == 1
    for route in (tda.TDA_ROUTE_FACTORED, tda.TDA_ROUTE_MATERIALIZE):
        wsb = tda.tda_workspace_size(tda.TDA_OP_PROJECT, L, tda.TDA_BF16, n, 0, route)
        ws = torch.empty(max(wsb, 256), dtype=torch.uint8, device=dev)
        phi = torch.full((n, k * k), float("nan"), device=dev)
        tda.tda_project(L, tda.TDA_BF16, Ad, Bd, n, phi, k * k, route, ws, wsb)
        tda.tda_device_status()
        got = phi.cpu().numpy()
        for e in range(n):
            assert rel_fro(got[e], ref[e]) <= TOL, (route, e)


def test_overlapped_query_side_matches_serial(dev):
    # the query side on a second stream beside an SM-capped train projection: same calls,
    # same arithmetic, so the features, preconditioned queries, scores and top-k are bit-identical
    linears, T, k, N, Nq = LLAMA1B, 256, 32, 1024, 16
    sb = math.sqrt(1e-3)
    At, Bt, Aq, Bq = [], [], [], []
    for li, (di, do) in enumerate(linears):
        At.append(fill(N, T, di, synth.SEED_A, li, 1.0, 0, 0.01, 0, dev))
        Bt.append(fill(N, T, do, synth.SEED_B, li, sb, 0, 0.01, 0, dev))
        Aq.append(fill(Nq, T, di, synth.SEED_A, li + synth.QUERY_STREAM_OFFSET, 1.0, 0, 0.01, 1000, dev))
        Bq.append(fill(Nq, T, do, synth.SEED_B, li + synth.QUERY_STREAM_OFFSET, sb, 0, 0.01, 1000, dev))
    out = []
    for overlap in (0, 24):
        pipe = BlockPipeline(linears, T, k, N, Nq, topk=50, precondition=True, lambda_rel=1e-2, device=dev)
        pipe.run(lambda li, L, r, phi, ld: tda.tda_project(L, tda.TDA_BF16, At[li], Bt[li], N, phi, ld, r),
                 lambda li, L, r, phi, ld: tda.tda_project(L, tda.TDA_BF16, Aq[li], Bq[li], Nq, phi, ld, r),
                 overlap_sms=overlap)
        tda.tda_device_status()
        out.append([x.cpu().numpy() for x in (pipe.Phi, pipe.Q, pipe.Qh, pipe.S, pipe.idx, pipe.val)])
        assert tda.tda_get_sm_budget() == 0
    for a, b in zip(*out):
        np.testing.assert_array_equal(a, b)
