"""One attribution pass over a block of linear layers, through the C ABI.

A transformer block's linears (e.g. q, k, v, o, gate, up, down) share the token
count T and the projection size k. For a batch of train and query examples the
pass is: route choice per linear (Sec. 3.2 / App. A.4 cost model), factored
projection of every example through every linear (Eq. 2), the per-linear Fisher
fit and damped inverse applied to the queries (App. B.2, B.3) -- the full empirical
Fisher of the projected features, or K-FAC / EK-FAC on the projected factors with
the covariances accumulated by the projection kernel itself -- the query x train
score matrix summed over the linears (Eq. 4's left side) and the top-k train
indices per query. Every step is a libtda.so call; this class only owns the
device buffers and the order of the calls.

Feature layout: linear l's k*k features of an example sit at columns
[l*k*k, (l+1)*k*k) of one row, so the preconditioner handles all linears in one
batched call and the score is one GEMM over all features.
"""
from __future__ import annotations

import torch

import paper_2609_38767_gb300 as tda
from paper_2609_38767_gb300 import shard


class BlockPipeline:
    CURVATURES = ("fisher", "kfac", "ekfac")

    def __init__(self, linears, T, k, n_train, n_query, *, topk=100, precondition=True,
                 lambda_abs=0.0, lambda_rel=1e-2, seed=0, layer0=0, device="cuda", curvature="fisher",
                 query_streams=8):
        assert curvature in self.CURVATURES
        self.query_streams = query_streams
        self.layers = [tda.LayerDesc(di, do, T, k, k, seed=seed, layer=layer0 + i)
                       for i, (di, do) in enumerate(linears)]
        self.N, self.Nq, self.D = n_train, n_query, k * k
        self.nl = len(self.layers)
        self.DT = self.D * self.nl
        self.topk, self.precondition, self.curvature = topk, precondition, curvature
        self.lambda_abs, self.lambda_rel = lambda_abs, lambda_rel
        dev = torch.device(device)
        self.Phi = torch.empty((n_train, self.DT), dtype=torch.float32, device=dev)
        self.Q = torch.empty((n_query, self.DT), dtype=torch.float32, device=dev)
        self.Qh = torch.empty((n_query, self.DT), dtype=torch.float32, device=dev)
        self.S = torch.empty((n_query, n_train), dtype=torch.float32, device=dev)
        self.idx = torch.empty((n_query, topk), dtype=torch.int32, device=dev)
        self.val = torch.empty((n_query, topk), dtype=torch.float32, device=dev)
        self.k = k
        if curvature == "fisher":
            per = tda.tda_precondition_state_bytes(self.D, tda.TDA_F32)
            self.state = torch.empty(self.nl * per, dtype=torch.uint8, device=dev)
        else:
            self.kf_per = tda.tda_kfac_state_bytes(k, k)
            self.kf_states = torch.empty(self.nl * self.kf_per, dtype=torch.uint8, device=dev)
            self.kf_state = [self.kf_states[i * self.kf_per:(i + 1) * self.kf_per] for i in range(self.nl)]
            self.kf_wsb = max(tda.tda_kfac_workspace_size(L, tda.TDA_BF16) for L in self.layers)
            self.kf_ws = torch.empty(self.kf_wsb, dtype=torch.uint8, device=dev)

    def project_train_kfac(self, li, A, B, phi, ld):
        """Train projection of linear li that also accumulates its K-FAC factor covariances."""
        tda.tda_project_kfac(self.layers[li], tda.TDA_BF16, A, B, self.N, phi, ld, self.kf_state[li], self.kf_ws,
                             self.kf_wsb)

    def routes(self):
        return [tda.tda_route(L, tda.TDA_OP_PROJECT, self.N, 0, tda.TDA_BF16)[0] for L in self.layers]

    def run(self, project_train, project_query, after_train_linear=None, mark=None, overlap_sms=0, dist=None):
        """project_train(li, L, route, phi_view, ld) fills train features of linear li;
        project_query likewise for the queries. after_train_linear(li) is called after
        each train projection; mark(name) before each phase and mark(None) at the end
        (e.g. to record timing events on the stream).

        overlap_sms > 0 (Fisher curvature): the query side runs on a second stream
        beside the train projections, which leave that many SMs free
        (tda_set_sm_budget): the query projections first, then, as soon as linear
        l's train features exist, its Fisher fit, factorisation and preconditioning.
        The arithmetic of every call is unchanged, so are the results.

        dist (torch.distributed, train examples sharded over its ranks): the curvature is
        fitted over all shards -- the sums are all-reduced before the factorisation and
        every rank preconditions its queries with the same global curvature."""
        mark = mark or (lambda name: None)
        world = dist.get_world_size() if dist is not None else 1
        if overlap_sms > 0 and self.precondition and self.curvature == "fisher" and world == 1:
            return self._run_overlapped(project_train, project_query, after_train_linear, mark, overlap_sms)
        routes = self.routes()
        D, DT = self.D, self.DT
        kfac = self.precondition and self.curvature != "fisher"
        if kfac:
            tda.tda_kfac_reset(self.k, self.k, self.kf_states, n_layers=self.nl)
        mark("project_train")
        for li, L in enumerate(self.layers):
            project_train(li, L, routes[li], self.Phi[:, li * D:], DT)
            if after_train_linear:
                after_train_linear(li)
        mark("project_query")
        self._project_queries(project_query, routes)
        target = self.Q
        if kfac:
            k = self.k
            nl, sts = self.nl, self.kf_states
            if world > 1:
                mark("curvature_allreduce")
                shard.allreduce_kfac(sts, nl, k, k, self.kf_per, dist, world)
            mark("kfac_eigen")
            tda.tda_kfac_eigen(k, k, sts, n_layers=nl)
            if self.curvature == "ekfac":
                mark("ekfac_eigenvalues")
                tda.tda_kfac_accumulate_eigenvalues(k, k, sts, self.Phi, self.N, DT, self.kf_ws, self.kf_wsb,
                                                    n_layers=nl)
                if world > 1:
                    shard.allreduce_kfac(sts, nl, k, k, self.kf_per, dist, world, eigenvalue_sums=True)
            mark("apply")
            kind = tda.TDA_EKFAC if self.curvature == "ekfac" else tda.TDA_KFAC
            tda.tda_kfac_apply(kind, k, k, sts, self.lambda_abs, self.lambda_rel, self.Q, self.Nq, DT, self.Qh, DT,
                               n_layers=nl)
            target = self.Qh
        elif self.precondition:
            nl, st, f32 = self.nl, self.state, tda.TDA_F32
            mark("fisher_fit")
            tda.tda_precondition(tda.TDA_PC_RESET, nl, D, f32, st)
            tda.tda_precondition(tda.TDA_PC_FIT_ACCUM, nl, D, f32, st, phi=self.Phi, n=self.N, ld_phi=DT)
            if world > 1:
                mark("curvature_allreduce")
                shard.allreduce_fisher(st, nl, D, tda.tda_precondition_state_bytes(D, f32), 4, dist, world)
            mark("factor_apply")
            tda.tda_precondition(tda.TDA_PC_FACTOR_APPLY, nl, D, f32, st, n_total=self.N * world,
                                 lambda_abs=self.lambda_abs, lambda_rel_mean_eig=self.lambda_rel,
                                 q=self.Q, n_q=self.Nq, ld_q=DT, qhat=self.Qh, ld_qhat=DT)
            target = self.Qh
        self._score(target, mark)

    def _project_queries(self, project_query, routes):
        """The query projections of all linears. A query batch is smaller than the GPU (64
        examples fill 128 of 152 SMs), so the linears go out on query_streams streams at once
        and the later launches fill the SMs the earlier ones leave idle; every launch writes
        its own feature columns, so the results do not depend on the order."""
        D, DT = self.D, self.DT
        n = min(self.query_streams, self.nl)
        if n <= 1 or not torch.cuda.is_available():
            for li, L in enumerate(self.layers):
                project_query(li, L, routes[li], self.Q[:, li * D:], DT)
            return
        main = torch.cuda.current_stream()
        if len(getattr(self, "_qstreams", ())) < n:
            self._qstreams = [torch.cuda.Stream(device=main.device) for _ in range(n)]
        streams = self._qstreams[:n]
        for s in streams:
            s.wait_stream(main)
        for li, L in enumerate(self.layers):
            with torch.cuda.stream(streams[li % n]):
                project_query(li, L, routes[li], self.Q[:, li * D:], DT)
        for s in streams:
            main.wait_stream(s)

    def _score(self, target, mark):
        DT = self.DT
        mark("score")
        tda.tda_score(target, tda.TDA_F32, self.Nq, DT, self.Phi, self.N, DT, DT, self.S, self.N, 0.0)
        mark("topk")
        tda.tda_topk(self.S, self.Nq, self.N, self.N, self.topk, self.idx, self.val)
        mark(None)

    def _run_overlapped(self, project_train, project_query, after_train_linear, mark, overlap_sms):
        routes = self.routes()
        D, DT, f32 = self.D, self.DT, tda.TDA_F32
        per = tda.tda_precondition_state_bytes(D, f32)
        main = torch.cuda.current_stream()
        if getattr(self, "_side", None) is None:
            self._side = torch.cuda.Stream(device=main.device)
        side = self._side
        sms = torch.cuda.get_device_properties(main.device).multi_processor_count
        side.wait_stream(main)  # inputs written on the main stream
        with torch.cuda.stream(side):
            for li, L in enumerate(self.layers):
                project_query(li, L, routes[li], self.Q[:, li * D:], DT)
        budget = tda.tda_get_sm_budget()
        tda.tda_set_sm_budget(max(1, sms - overlap_sms))
        try:
            mark("project_train")
            for li, L in enumerate(self.layers):
                project_train(li, L, routes[li], self.Phi[:, li * D:], DT)
                if after_train_linear:
                    after_train_linear(li)
                done = torch.cuda.Event()
                done.record(main)
                side.wait_event(done)
                with torch.cuda.stream(side):
                    st = self.state[li * per:(li + 1) * per]
                    tda.tda_precondition(tda.TDA_PC_RESET, 1, D, f32, st)
                    tda.tda_precondition(tda.TDA_PC_FIT_ACCUM, 1, D, f32, st, phi=self.Phi[:, li * D:], n=self.N,
                                         ld_phi=DT)
                    tda.tda_precondition(tda.TDA_PC_FACTOR_APPLY, 1, D, f32, st, n_total=self.N,
                                         lambda_abs=self.lambda_abs, lambda_rel_mean_eig=self.lambda_rel,
                                         q=self.Q[:, li * D:], n_q=self.Nq, ld_q=DT, qhat=self.Qh[:, li * D:],
                                         ld_qhat=DT)
        finally:
            tda.tda_set_sm_budget(budget)
        mark("query_side_tail")
        main.wait_stream(side)
        self._score(self.Qh, mark)
