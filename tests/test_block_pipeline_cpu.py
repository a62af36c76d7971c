"""Host logic of one attribution pass over a block (BlockPipeline), on the CPU.

BlockPipeline owns the block's buffers and orders the library calls: each
linear's features in its own k*k columns of one row per example, one batched
Fisher fit and damped inverse over all linears, one score over all features,
the top-k. With a recording fake in place of the library calls (and the route
cost model of the real library, which is host-only), the pass is compared with
the block computed directly with the oracle: per-linear Fisher, damping
relative to the mean eigenvalue, damped inverse on the queries, score summed
over the linears, top-k -- and, without the preconditioner, GradDot scores.
"""
import numpy as np
import pytest
import torch

import paper_2609_38767_gb300 as tda
from paper_2609_38767_gb300 import build as tbuild
from paper_2609_38767_gb300 import synth

from fake_tda import FakeLib, install, pipeline_class

BlockPipeline = pipeline_class("block", "BlockPipeline")

LIN = [(32, 16), (16, 48), (24, 24)]
T, K, N, NQ, TOPK = 7, 4, 48, 5, 6


def factors():
    out = []
    for li, (di, do) in enumerate(LIN):
        out.append(tuple(synth.to_f64(x, "bf16") for x in (
            synth.factors(synth.SEED_A, li, N, T, di, 1.0, dtype="bf16", mask_p=0.1),
            synth.factors(synth.SEED_B, li, N, T, do, 0.1, dtype="bf16", mask_p=0.1),
            synth.factors(synth.SEED_A, li + synth.QUERY_STREAM_OFFSET, NQ, T, di, 1.0, dtype="bf16"),
            synth.factors(synth.SEED_B, li + synth.QUERY_STREAM_OFFSET, NQ, T, do, 0.1, dtype="bf16"))))
    return out


@pytest.mark.parametrize("precondition", [True, False])
def test_block_pipeline_order_and_layout_match_oracle(orc, monkeypatch, precondition):
    tbuild.build()  # the route cost model is the real library's (host-only)
    fake = FakeLib(orc)
    install(fake, monkeypatch)
    f = factors()
    D = K * K
    pipe = BlockPipeline(LIN, T, K, N, NQ, topk=TOPK, precondition=precondition, lambda_rel=1e-2, device="cpu",
                         layer0=3)
    for t in (pipe.Phi, pipe.Q, pipe.Qh, pipe.S):
        t.fill_(float("nan"))
    written = []

    def project(role):
        def run(li, L, route, phi, ld):
            assert L.layer == 3 + li and ld == pipe.DT == phi.stride(0)
            assert route in (tda.TDA_ROUTE_FACTORED, tda.TDA_ROUTE_MATERIALIZE)
            A, B = (f[li][0], f[li][1]) if role == "train" else (f[li][2], f[li][3])
            x = orc.project(A, B, K, K, 0, L.layer).reshape(A.shape[0], D)
            phi[:, :D] = torch.from_numpy(x)
            written.append((role, li, phi.data_ptr()))
        return run

    marks = []
    pipe.run(project("train"), project("query"), mark=marks.append)

    # each linear wrote its own D columns of the shared rows
    base = {"train": pipe.Phi.data_ptr(), "query": pipe.Q.data_ptr()}
    assert [(r, li) for r, li, _ in written] == [("train", i) for i in range(3)] + [("query", i) for i in range(3)]
    assert all(p == base[r] + 4 * li * D for r, li, p in written)
    phases = ["project_train", "project_query"] + (["fisher_fit", "factor_apply"] if precondition else [])
    assert marks == phases + ["score", "topk", None]

    phi = np.concatenate([orc.project(a, b, K, K, 0, 3 + li).reshape(N, D) for li, (a, b, _, _) in enumerate(f)], 1)
    q = np.concatenate([orc.project(a, b, K, K, 0, 3 + li).reshape(NQ, D) for li, (_, _, a, b) in enumerate(f)], 1)
    if precondition:
        qh = np.empty_like(q)
        for li in range(len(LIN)):
            F = orc.fisher(np.ascontiguousarray(phi[:, li * D:(li + 1) * D]))
            qh[:, li * D:(li + 1) * D] = orc.precondition(F, orc.damping(F, 0.0, 1e-2),
                                                          np.ascontiguousarray(q[:, li * D:(li + 1) * D]))
        fits = [c for c in fake.log if c[0] == "fit"]
        assert fits == [("fit", pipe.Phi.data_ptr(), len(LIN), N)]  # one batched call over all linears
    else:
        qh = q
        assert not [c for c in fake.log if c[0] in ("fit", "factor_apply")]
    S = orc.score(qh, phi)
    rel = float(np.linalg.norm(pipe.S.double().numpy() - S) / np.linalg.norm(S))
    assert rel <= 1e-5, rel  # fp32 buffers, as on the device
    oi, _ = orc.topk(S, TOPK)
    np.testing.assert_array_equal(pipe.idx.numpy(), oi)
