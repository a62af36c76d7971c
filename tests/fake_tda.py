"""A recording stand-in for the libtda calls that the host-side pipelines make
(StackJob, BlockPipeline), in fp64 numpy on the CPU, so that their order of
calls, buffers and shares can be tested without a GPU. Features come from the
oracle's projection; the Fisher fit, damped inverse, score and top-k are the
plain definitions. Test infrastructure only."""
import contextlib

import numpy as np
import torch

import paper_2609_38767_gb300 as tda
from paper_2609_38767_gb300 import synth


def bf16_tensor(bits):
    return torch.from_numpy(bits.view(np.int16)).view(torch.bfloat16)


def to64(x):
    return synth.to_f64(x.view(torch.int16).numpy().view(np.uint16), "bf16")


class FakeLib:
    """The library calls StackJob makes, in fp64 on the CPU, with a log of each call."""

    def __init__(self, orc):
        self.orc = orc
        self.log = []
        self.states = {}

    def tda_precondition_state_bytes(self, D, dtype):
        return 64

    def tda_project_host(self, L, dtype, A, B, n, phi, ld, ws, wsb, stream=None):
        assert dtype == tda.TDA_BF16 and ld == phi.stride(0)
        f = self.orc.project(to64(A), to64(B), L.k_in, L.k_out, L.seed, L.layer).reshape(n, -1)
        phi[:n, :f.shape[1]] = torch.from_numpy(f)
        self.log.append(("project", L.layer, phi.data_ptr(), n))

    def tda_precondition(self, op, nl, D, dtype, st, phi=None, n=0, ld_phi=0, n_total=0, lambda_abs=0.0,
                         lambda_rel_mean_eig=0.0, q=None, n_q=0, ld_q=0, qhat=None, ld_qhat=0, stream=None):
        key = st.data_ptr()
        if op == tda.TDA_PC_RESET:
            self.states[key] = [np.zeros((D, D)) for _ in range(nl)]
        elif op == tda.TDA_PC_FIT_ACCUM:
            for l in range(nl):
                Pl = phi[:n, l * D:(l + 1) * D].double().numpy()
                self.states[key][l] += Pl.T @ Pl
            self.log.append(("fit", phi.data_ptr(), nl, n))
        elif op == tda.TDA_PC_FACTOR_APPLY:
            for l in range(nl):
                F = self.states[key][l] / n_total
                lam = lambda_abs + lambda_rel_mean_eig * np.trace(F) / D
                Ql = q[:n_q, l * D:(l + 1) * D].double().numpy()
                qhat[:n_q, l * D:(l + 1) * D] = torch.from_numpy(np.linalg.solve(F + lam * np.eye(D), Ql.T).T)
            self.log.append(("factor_apply", q.data_ptr(), nl))
        else:
            raise AssertionError(op)

    def tda_score(self, Qh, qdt, n_q, ld_q, Phi, n_t, ld_phi, D, S, ld_S, beta=0.0, stream=None):
        prod = Qh[:n_q, :D].double() @ Phi[:n_t, :D].double().T
        S[:n_q, :n_t] = (prod if beta == 0.0 else beta * S[:n_q, :n_t].double() + prod).float()
        self.log.append(("score", S.data_ptr(), Phi.data_ptr(), D, beta))

    def tda_topk(self, S, n_q, n_t, ld_S, k, idx, val=None, stream=None):
        oi, ov = self.orc.topk(S[:n_q, :n_t].double().numpy(), k)
        idx[:n_q] = torch.from_numpy(oi.astype(np.int32))
        val[:n_q] = torch.from_numpy(ov.astype(np.float32))
        self.log.append(("topk", S.data_ptr(), n_q))


def install(fake, monkeypatch, cuda_streams=False):
    """Put the fake's calls in place of the binding's; cuda_streams: also stand in for the
    current-stream context that StackJob's in-line query side re-enters."""
    for name in ("tda_precondition_state_bytes", "tda_project_host", "tda_precondition", "tda_score", "tda_topk"):
        monkeypatch.setattr(tda, name, getattr(fake, name))
    if cuda_streams:
        monkeypatch.setattr(torch.cuda, "current_stream", lambda *a, **k: None)
        monkeypatch.setattr(torch.cuda, "stream", lambda s: contextlib.nullcontext())


def pipeline_class(module, name):
    """The host pipeline class `name` of paper_2609_38767_gb300.<module>, or, when the
    environment names another source for that module (TDA_<MODULE>_SOURCE; the mutation
    test of the host-logic tests plants mistakes in a copy), the class from that copy."""
    import importlib
    import importlib.util
    import os

    src = os.environ.get(f"TDA_{module.upper()}_SOURCE")
    if not src:
        return getattr(importlib.import_module(f"paper_2609_38767_gb300.{module}"), name)
    spec = importlib.util.spec_from_file_location(f"{module}_variant", src)
    mod = importlib.util.module_from_spec(spec)
    spec.loader.exec_module(mod)
    return getattr(mod, name)
