"""The streamed stack job (software-pipelined chunks) against the oracle.

Three jobs run back to back on a small stack of six linears (three layers of
two), each job's training set drawn from its own windows of a factor pool, in
chunks. After the third job, the score matrix of the second job and the top-k of
the first are complete; both are compared with the oracle's fp64 features,
Fisher, damped inverse (Woodbury form: fewer examples than features), score
matrix and top-k over the same factors. The shares of the query side differ in
size (six linears over four steps), D = 4096 takes the blocked tensor-core
preconditioner, and the train projections of a chunk run on one, two or three
streams, the query side in line, on a stream of its own, or enqueued by a host
thread of its own with its bulk kernels on a third stream.
"""
import os

import numpy as np
import pytest
import torch

import paper_2609_38767_gb300 as tda
from paper_2609_38767_gb300 import build as tbuild
from paper_2609_38767_gb300 import synth
from paper_2609_38767_gb300.stream import StackJob

pytestmark = pytest.mark.gpu
TOL = 2e-2
LIN = [(512, 256), (256, 512)] * 3
T, K, N, CHUNK, NQ, TOPK, P, PQ = 32, 64, 64, 16, 8, 5, 24, 11


def rel_fro(x, ref):
    x, ref = np.asarray(x, np.float64), np.asarray(ref, np.float64)
    return float(np.linalg.norm(x - ref) / np.linalg.norm(ref))


def pools():
    # host copies (for the oracle) and device copies of the factor pools, one pool per linear
    out = []
    for li, (di, do) in enumerate(LIN):
        A = synth.factors(synth.SEED_A, li, P, T, di, 1.0, dtype="bf16", mask_p=0.05)
        B = synth.factors(synth.SEED_B, li, P, T, do, 0.03, dtype="bf16", mask_p=0.05)
        Aq = synth.factors(synth.SEED_A, li + synth.QUERY_STREAM_OFFSET, PQ, T, di, 1.0, dtype="bf16")
        Bq = synth.factors(synth.SEED_B, li + synth.QUERY_STREAM_OFFSET, PQ, T, do, 0.03, dtype="bf16")
        out.append((A, B, Aq, Bq))
    return out


def window(role, li, j, s):
    """Pool rows of (role, linear, job, chunk): a window that wraps around the pool."""
    if role == "train":
        return [(7 * j + 3 * s + 5 * li + r) % P for r in range(CHUNK)]
    return [(2 * j + li + r) % PQ for r in range(NQ)]


@pytest.mark.parametrize("train_streams,query_stream,opts", [
    (1, False, {}), (3, True, {}),
    # the query side enqueued by a host thread of its own, its bulk kernels on a third stream,
    # stream priorities train > factorisation chain > bulk
    (2, True, {"side_thread": True, "bulk_priority": 0, "train_priority": -1, "query_priority": -2})])
def test_stack_job_matches_oracle(orc, train_streams, query_stream, opts):
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    tbuild.build()
    tda.load()
    dev = torch.device("cuda:0")
    host = pools()
    to = lambda x: torch.from_numpy(x.view(np.int16)).view(torch.bfloat16).to(dev)
    devp = [tuple(to(x) for x in p) for p in host]

    def factors(role, li, j, s):
        rows = window(role, li, j, s)
        A, B = (devp[li][0], devp[li][1]) if role == "train" else (devp[li][2], devp[li][3])
        pieces, r = [], 0
        while r < len(rows):  # contiguous runs of pool rows
            e = r
            while e + 1 < len(rows) and rows[e + 1] == rows[e] + 1:
                e += 1
            pieces.append((A[rows[r]:rows[e] + 1], B[rows[r]:rows[e] + 1], r, e - r + 1))
            r = e + 1
        return pieces

    job = StackJob(LIN, T, K, N, CHUNK, NQ, topk=TOPK, lambda_rel=1e-2, device=dev, train_streams=train_streams,
                   query_stream=query_stream, **opts)
    marks = []
    for j in range(3):
        for s in range(job.C):
            job.step(j, s, factors, mark=marks.append)
    job.join()
    job.close()
    torch.cuda.synchronize()
    tda.tda_device_status()
    assert {"project_train", "fisher_fit", "project_query", "factor_apply", "score", "topk"} <= set(marks)

    orc.set_threads(os.cpu_count() or 1)
    D = K * K

    def oracle_job(j):
        phi = np.zeros((N, D * len(LIN)))
        q = np.zeros((NQ, D * len(LIN)))
        for li in range(len(LIN)):
            A, B, Aq, Bq = host[li]
            for s in range(job.C):
                rows = window("train", li, j, s)
                f = orc.project(synth.to_f64(A[rows], "bf16"), synth.to_f64(B[rows], "bf16"), K, K, 0, li)
                phi[s * CHUNK:(s + 1) * CHUNK, li * D:(li + 1) * D] = f.reshape(CHUNK, D)
            rows = window("query", li, j, 0)
            q[:, li * D:(li + 1) * D] = orc.project(synth.to_f64(Aq[rows], "bf16"), synth.to_f64(Bq[rows], "bf16"),
                                                    K, K, 0, li).reshape(NQ, D)
        qh = np.empty_like(q)
        for li in range(len(LIN)):
            P_ = np.ascontiguousarray(phi[:, li * D:(li + 1) * D])
            lam = orc.damping_features(P_, 0.0, 1e-2)
            qh[:, li * D:(li + 1) * D] = orc.precondition_lowrank(P_, lam, np.ascontiguousarray(q[:, li * D:(li + 1) * D]))
        return phi, orc.score(qh, phi)

    phi1, S1 = oracle_job(1)
    assert rel_fro(job.Phi[1].cpu().numpy(), phi1) <= TOL
    assert rel_fro(job.S[1].cpu().numpy(), S1) <= TOL
    _, S0 = oracle_job(0)
    S0_gpu = job.S[0].cpu().numpy()
    assert rel_fro(S0_gpu, S0) <= TOL
    # job 0's top-k, taken during job 2: bit-exact selection on the GPU's own job-0 scores
    oi, ov = orc.topk(S0_gpu.astype(np.float64), TOPK)
    np.testing.assert_array_equal(job.idx.cpu().numpy(), oi)
    np.testing.assert_array_equal(job.val.cpu().numpy(), ov.astype(np.float32))
