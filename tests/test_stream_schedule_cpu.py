"""Host logic of the streamed stack job (StackJob), on the CPU.

StackJob only orders libtda calls: which chunk a step projects into which
feature rows, which share of linears of which job's query side it fits,
factors and scores, into which of the double-buffered feature and score
matrices, and which job's top-k it takes. This test runs that order without a
GPU by standing a recording fake in for the library calls (fp64 numpy; the
oracle's projection for the features), runs three jobs back to back and checks:

* every job's score matrix equals the whole-job computation done directly with
  the oracle (Fisher over the job's full training set, damping relative to the
  mean eigenvalue, damped inverse on the queries, score) -- so no share reads
  another job's features or a stale score buffer;
* job 0's top-k, taken during job 2, is the oracle's top-k of job 0's scores;
* each step does exactly its share: one chunk per linear, the s-th of C
  near-equal shares of the previous job's linears, the s-th share of the query
  rows of the job before.

The library itself is exercised against the oracle on the GPU in
test_gpu_stream.py; here only the schedule is under test.
"""
import numpy as np
import pytest

from paper_2609_38767_gb300 import synth
from fake_tda import FakeLib, bf16_tensor, install, pipeline_class

StackJob = pipeline_class("stream", "StackJob")

LIN = [(24, 16), (16, 40), (32, 24), (24, 24), (40, 16)]  # five linears over four steps: shares 1, 1, 1, 2
T, K, N, CHUNK, NQ, TOPK, P, PQ = 6, 4, 64, 16, 6, 5, 40, 9
LAM_REL = 1e-2


def window(role, li, j, s):
    if role == "train":
        return [(11 * j + 5 * s + 3 * li + r) % P for r in range(CHUNK)]
    return [(2 * j + li + r) % PQ for r in range(NQ)]


@pytest.fixture
def fake(orc, monkeypatch):
    f = FakeLib(orc)
    install(f, monkeypatch, cuda_streams=True)  # the in-line query side re-enters the current stream
    return f


def pools():
    out = []
    for li, (di, do) in enumerate(LIN):
        A = synth.factors(synth.SEED_A, li, P, T, di, 1.0, dtype="bf16", mask_p=0.1)
        B = synth.factors(synth.SEED_B, li, P, T, do, 0.1, dtype="bf16", mask_p=0.1)
        Aq = synth.factors(synth.SEED_A, li + synth.QUERY_STREAM_OFFSET, PQ, T, di, 1.0, dtype="bf16")
        Bq = synth.factors(synth.SEED_B, li + synth.QUERY_STREAM_OFFSET, PQ, T, do, 0.1, dtype="bf16")
        out.append((A, B, Aq, Bq))
    return out


def test_stack_job_schedule_matches_whole_job_oracle(orc, fake):
    host = pools()

    def factors(role, li, j, s):
        A, B = (host[li][0], host[li][1]) if role == "train" else (host[li][2], host[li][3])
        rows = window(role, li, j, s)
        return [(bf16_tensor(A[rows]), bf16_tensor(B[rows]), 0, len(rows))]

    job = StackJob(LIN, T, K, N, CHUNK, NQ, topk=TOPK, lambda_rel=LAM_REL, device="cpu", proj_ws=False)
    assert job.C == 4 and [job.share(s, len(LIN)) for s in range(4)] == [(0, 1), (1, 2), (2, 3), (3, 5)]
    for t in (job.Phi[0], job.Phi[1], job.S[0], job.S[1], job.Q, job.Qh):
        t.fill_(float("nan"))  # anything read before it is written shows up in the scores
    per_step = []
    for j in range(3):
        for s in range(job.C):
            n0 = len(fake.log)
            job.step(j, s, factors)
            per_step.append((j, s, fake.log[n0:]))

    D, DT = K * K, K * K * len(LIN)

    def oracle_job(j):
        phi = np.zeros((N, DT))
        q = np.zeros((NQ, DT))
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
            F = orc.fisher(np.ascontiguousarray(phi[:, li * D:(li + 1) * D]))
            lam = orc.damping(F, 0.0, LAM_REL)
            qh[:, li * D:(li + 1) * D] = orc.precondition(F, lam, np.ascontiguousarray(q[:, li * D:(li + 1) * D]))
        return phi, orc.score(qh, phi)

    rel = lambda x, ref: float(np.linalg.norm(np.asarray(x, np.float64) - ref) / np.linalg.norm(ref))
    phi2, _ = oracle_job(2)
    phi1, S1 = oracle_job(1)
    _, S0 = oracle_job(0)
    # fp32 buffers (as on the device): features and scores to fp32 rounding
    assert rel(job.Phi[0].numpy(), phi2) <= 1e-6  # job 2 overwrote job 0's features, after job 0's query side
    assert rel(job.Phi[1].numpy(), phi1) <= 1e-6
    assert rel(job.S[1].numpy(), S1) <= 1e-5  # job 1's scores, completed during job 2
    assert rel(job.S[0].numpy(), S0) <= 1e-5  # job 0's scores, completed during job 1
    oi, ov = orc.topk(job.S[0].double().numpy(), TOPK)
    np.testing.assert_array_equal(job.idx.numpy(), oi)
    oi_ref, _ = orc.topk(S0, TOPK)
    np.testing.assert_array_equal(job.idx.numpy(), oi_ref)

    # each step does exactly its share of each phase
    Phi_ptr = [job.Phi[b].data_ptr() for b in range(2)]
    S_ptr = [job.S[b].data_ptr() for b in range(2)]
    for j, s, calls in per_step:
        proj = [c for c in calls if c[0] == "project"]
        train = [c for c in proj if c[2] - Phi_ptr[j % 2] in range(0, N * DT * 4)]
        assert [c[1] for c in train] == list(range(len(LIN))) and all(c[3] == CHUNK for c in train)
        for c in train:  # chunk s's rows of linear c[1]'s columns
            assert c[2] == Phi_ptr[j % 2] + 4 * (s * CHUNK * DT + c[1] * D)
        l0, l1 = job.share(s, len(LIN))
        fits = [c for c in calls if c[0] == "fit"]
        scores = [c for c in calls if c[0] == "score"]
        topks = [c for c in calls if c[0] == "topk"]
        if j >= 1:  # share s of job j-1's query side, on job j-1's buffers
            b = (j - 1) % 2
            assert fits == [("fit", Phi_ptr[b] + 4 * l0 * D, l1 - l0, N)]
            assert [c[1] for c in proj if c not in train] == list(range(l0, l1))
            assert scores == [("score", S_ptr[b], Phi_ptr[b] + 4 * l0 * D, (l1 - l0) * D, 0.0 if l0 == 0 else 1.0)]
        else:
            assert not fits and not scores and len(proj) == len(LIN)
        r0, r1 = job.share(s, NQ)
        if j >= 2:  # share s of job j-2's query rows
            assert topks == [("topk", S_ptr[(j - 2) % 2] + 4 * r0 * N, r1 - r0)]
        else:
            assert not topks
