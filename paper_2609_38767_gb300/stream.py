"""A streamed attribution job over a stack of layers, through the C ABI.

The training set of a job is too large to hold its factors, so it streams in
chunks (App. A.2: the factors are projected as they arrive and never buffered
whole); the projected features stay resident. A job over N_train examples and
a stack of linears is, per linear (Sec. 3.2, App. B.2, B.3):

  project every training chunk (Eq. 2) into the resident features, fit the
  linear's Fisher F = Phi^T Phi / N over all of them, project the queries,
  factor F + lambda I and precondition the queries (lambda = lambda_rel x mean
  eigenvalue), add the linear's share of the query x train score matrix
  (Eq. 4's left side), and finally take the top-k train indices per query.

Jobs run back to back, software-pipelined in steps of one chunk: step s of job
j projects chunk s of job j; it also runs the s-th share of job j-1's query
side (the linears in [s L / C, (s+1) L / C) of L linears: their Fisher fit over
job j-1's features, query projections, factorisation and preconditioning, and
their share of job j-1's score), and the top-k of the s-th share of job j-2's
query rows (C chunks per job). Each step thus does 1/C of every phase of a job,
and C consecutive steps do a whole job's work. Buffers that two jobs in flight
need at once (features, score matrix) are double-buffered by job parity; the
Fisher states hold one share of linears.

Every step is a libtda.so call; this class only owns the device buffers and the
order of the calls. The caller provides the factors of a (role, linear, chunk)
as pieces (device tensors, or pinned host tensors for tda_project_host).
"""
from __future__ import annotations

import queue
import threading

import torch

import paper_2609_38767_gb300 as tda


class StackJob:
    def __init__(self, linears, T, k, n_train, chunk, n_query, *, topk=100, lambda_rel=1e-2, lambda_abs=0.0,
                 seed=0, device="cuda", host_ws_bytes=0, train_streams=1, proj_ws=True, query_stream=False,
                 query_priority=0, balance=True, train_priority=0, bulk_priority=None, side_thread=False):
        """linears: [(d_in, d_out)] of the whole stack, in layer order (linear i uses projection
        layer id i). n_train must be a multiple of chunk. train_streams > 1 spreads the train
        projections of a chunk round-robin over that many streams, so that a launch's CTAs fill
        the SMs its predecessor's last tiles leave idle (every launch writes its own feature
        columns: the results do not depend on the order). proj_ws: give the factored projection
        its optional workspace (k = 128: precomputed sign tables). balance: let it use that
        workspace for balanced token-tile ranges too (otherwise every SM takes whole examples,
        whose staggered ends the next launch on another stream fills). query_stream: run the query
        side and the top-k on a stream of their own (priority query_priority), beside the
        next chunks' projections; events order the two job-boundary dependencies (a job's
        query side starts after its last chunk is projected; a job's features are overwritten
        two jobs later only after that query side has read them). train_priority: priority of
        the train projection streams. bulk_priority: with query_stream, run the query side's
        bulk kernels (Fisher fit and query projections) on a third stream of this priority,
        so that they can yield to the train projections while the latency-bound factorisation
        chain keeps query_priority (lower number = higher priority). side_thread: with
        query_stream, a host thread of its own enqueues the query side, so that a query-side
        stream that the GPU serves late (a full launch queue) cannot hold up the enqueueing of
        the next chunks' projections."""
        assert n_train % chunk == 0 and n_train >= topk >= 1
        self.layers = [tda.LayerDesc(di, do, T, k, k, seed=seed, layer=i) for i, (di, do) in enumerate(linears)]
        self.nl = len(self.layers)
        self.T, self.k, self.D = T, k, k * k
        self.DT = self.D * self.nl
        self.N, self.chunk, self.Nq, self.topk = n_train, chunk, n_query, topk
        self.C = n_train // chunk
        self.lambda_abs, self.lambda_rel = lambda_abs, lambda_rel
        dev = torch.device(device)
        self.per = tda.tda_precondition_state_bytes(self.D, tda.TDA_F32)
        self.Phi = [torch.empty((n_train, self.DT), dtype=torch.float32, device=dev) for _ in range(2)]
        self.share_max = max(b - a for a, b in (self.share(s, self.nl) for s in range(self.C)))
        self.state = torch.empty(max(self.share_max, 1) * self.per, dtype=torch.uint8, device=dev)
        self.S = [torch.empty((n_query, n_train), dtype=torch.float32, device=dev) for _ in range(2)]
        self.Q = torch.empty((n_query, self.DT), dtype=torch.float32, device=dev)
        self.Qh = torch.empty((n_query, self.DT), dtype=torch.float32, device=dev)
        self.idx = torch.empty((n_query, topk), dtype=torch.int32, device=dev)
        self.val = torch.empty((n_query, topk), dtype=torch.float32, device=dev)
        self.host_ws_bytes = host_ws_bytes
        self.host_ws = torch.empty(host_ws_bytes, dtype=torch.uint8, device=dev) if host_ws_bytes else None
        self.train_streams = max(1, train_streams)
        self._streams = []
        # one workspace per stream (a call writes its sign tables into it)
        self.proj_wsb = max(tda.tda_workspace_size(tda.TDA_OP_PROJECT, L, tda.TDA_BF16, chunk, 0,
                                                   tda.TDA_ROUTE_FACTORED) for L in self.layers) if proj_ws else 0
        if proj_ws and not balance:  # room for the k = 128 sign tables only
            self.proj_wsb = 2 * k * max(di + do for di, do in linears) if k == 128 else 0
        self.proj_ws = [torch.empty(self.proj_wsb, dtype=torch.uint8, device=dev)
                        for _ in range(self.train_streams + 1)] if self.proj_wsb else None
        self.side = torch.cuda.Stream(device=dev, priority=query_priority) if query_stream else None
        self.side_bulk = (torch.cuda.Stream(device=dev, priority=bulk_priority)
                          if query_stream and bulk_priority is not None else None)
        self.train_priority = train_priority
        self._dev = dev
        self._worker = None
        self._qd_ready = {}  # job -> threading.Event: its query_done event has been recorded
        if query_stream and side_thread:
            self._tasks = queue.Queue()
            self._err = None
            self._worker = threading.Thread(target=self._run_side, name="tda-query-side", daemon=True)
            self._worker.start()
        self._train_done = {}  # job -> event after its last chunk's projections (train stream)
        self._query_done = {}  # job -> event after its last query share (query stream)

    # ------------------------------------------------------------------ shares of a job
    def share(self, s, total):
        """[lo, hi) of `total` items handled at step s (the s-th of C near-equal shares)."""
        return total * s // self.C, total * (s + 1) // self.C

    def _project(self, L, pieces, phi, hook=None, li=0, role="train", slot=0):
        """pieces: [(A, B, row, n)] -- n examples written to feature row `row` of phi."""
        ws = self.proj_ws[slot] if self.proj_ws else None
        for A, B, row, n in pieces:
            if hook:
                hook(role, li, "begin", n)
            if A.is_cuda:
                tda.tda_project(L, tda.TDA_BF16, A, B, n, phi[row:], self.DT, tda.TDA_ROUTE_FACTORED, ws,
                                self.proj_wsb if ws is not None else 0)
            else:
                tda.tda_project_host(L, tda.TDA_BF16, A, B, n, phi[row:], self.DT, self.host_ws, self.host_ws_bytes)
            if hook:
                hook(role, li, "end", n)

    def train_part(self, j, s, factors, mark=None, hook=None):
        """Chunk s of job j: project it through every linear into the resident features."""
        if mark:
            mark("project_train")
        Phi = self.Phi[j % 2][s * self.chunk:(s + 1) * self.chunk]
        n = min(self.train_streams, self.nl)
        if n <= 1:
            for li, L in enumerate(self.layers):
                self._project(L, factors("train", li, j, s), Phi[:, li * self.D:], hook, li, "train")
            return
        main = torch.cuda.current_stream()
        if len(self._streams) < n:
            self._streams = [torch.cuda.Stream(device=main.device, priority=self.train_priority) for _ in range(n)]
        for st in self._streams[:n]:
            st.wait_stream(main)
        for li, L in enumerate(self.layers):
            with torch.cuda.stream(self._streams[li % n]):
                self._project(L, factors("train", li, j, s), Phi[:, li * self.D:], hook, li, "train", li % n)
        for st in self._streams[:n]:
            main.wait_stream(st)

    def query_part(self, j, s, factors, mark=None, hook=None):
        """Share s of job j's query side: the Fisher fit of linears [l0, l1) over all of job
        j's features, their query projections, factorisation and preconditioning, and their
        share of the score matrix."""
        b = j % 2
        mark = mark or (lambda name: None)
        l0, l1 = self.share(s, self.nl)
        if l1 == l0:
            return
        D, DT = self.D, self.DT
        st = self.state[:(l1 - l0) * self.per]
        slot = self.train_streams  # the query side's own projection workspace
        chain, bulk = torch.cuda.current_stream(), self.side_bulk
        if bulk is not None:
            bulk.wait_stream(chain)  # the previous share's factorisation is done with the state
        with torch.cuda.stream(bulk if bulk is not None else chain):
            mark("fisher_fit")
            tda.tda_precondition(tda.TDA_PC_RESET, l1 - l0, D, tda.TDA_F32, st)
            tda.tda_precondition(tda.TDA_PC_FIT_ACCUM, l1 - l0, D, tda.TDA_F32, st, phi=self.Phi[b][:, l0 * D:],
                                 n=self.N, ld_phi=DT)
            mark("project_query")
            for li in range(l0, l1):
                self._project(self.layers[li], factors("query", li, j, s), self.Q[:, li * D:], hook, li, "query",
                              slot)
            if bulk is not None:
                mark(None)
        if bulk is not None:
            chain.wait_stream(bulk)
        mark("factor_apply")
        tda.tda_precondition(tda.TDA_PC_FACTOR_APPLY, l1 - l0, D, tda.TDA_F32, st, n_total=self.N,
                             lambda_abs=self.lambda_abs, lambda_rel_mean_eig=self.lambda_rel, q=self.Q[:, l0 * D:],
                             n_q=self.Nq, ld_q=DT, qhat=self.Qh[:, l0 * D:], ld_qhat=DT)
        mark("score")
        tda.tda_score(self.Qh[:, l0 * D:], tda.TDA_F32, self.Nq, DT, self.Phi[b][:, l0 * D:], self.N, DT,
                      (l1 - l0) * D, self.S[b], self.N, 0.0 if l0 == 0 else 1.0)

    def topk_part(self, j, s, mark=None):
        """Share s of job j's query rows: their top-k train indices (job j's S is complete)."""
        r0, r1 = self.share(s, self.Nq)
        if r1 == r0:
            return
        if mark:
            mark("topk")
        tda.tda_topk(self.S[j % 2][r0:], r1 - r0, self.N, self.N, self.topk, self.idx[r0:], self.val[r0:])

    def _run_side(self):
        torch.cuda.set_device(self._dev)
        while True:
            task = self._tasks.get()
            try:
                if task is None:
                    return
                if self._err is None:
                    with torch.cuda.stream(self.side):
                        task()
            except BaseException as e:  # re-raised on the caller's thread by step() or join()
                self._err = e
                for ready in list(self._qd_ready.values()):
                    ready.set()  # a caller waiting for a job boundary wakes up and raises
            finally:
                self._tasks.task_done()

    def _side_part(self, j, s, factors, first_job, mark, hook, ready=None):
        """The query side of step s of job j, on the query-side stream (current stream);
        ready (threading.Event) is set once job j-1's query_done event is recorded."""
        if j - 1 >= first_job:
            if s == 0 and (j - 1) in self._train_done:
                self.side.wait_event(self._train_done.pop(j - 1))
            self.query_part(j - 1, s, factors, mark, hook)
            if s == self.C - 1:
                e = torch.cuda.Event()
                e.record(self.side)
                self._query_done[j - 1] = e
                if ready is not None:
                    ready.set()
        if j - 2 >= first_job:
            self.topk_part(j - 2, s, mark)
        if mark:
            mark(None)

    def step(self, j, s, factors, first_job=0, mark=None, hook=None):
        """Step s of job j: chunk s of job j, share s of job j-1's query side and of job
        j-2's top-k. Jobs before first_job do not exist (their shares are skipped)."""
        if self.side is None:
            self.train_part(j, s, factors, mark, hook)
            if j - 1 >= first_job:
                self.query_part(j - 1, s, factors, mark, hook)
            if j - 2 >= first_job:
                self.topk_part(j - 2, s, mark)
            if mark:
                mark(None)
            return
        main = torch.cuda.current_stream()
        if s == 0 and j - 2 >= first_job:
            ready = self._qd_ready.pop(j - 2, None)
            if ready is not None:
                ready.wait()  # the query-side thread has recorded job j-2's query_done
                if self._err is not None:
                    err, self._err = self._err, None
                    raise err
            if (j - 2) in self._query_done:
                main.wait_event(self._query_done.pop(j - 2))  # job j overwrites job j-2's features
        self.train_part(j, s, factors, mark, hook)
        if mark:
            mark(None)
        if s == self.C - 1:
            e = torch.cuda.Event()
            e.record(main)
            self._train_done[j] = e
        if self._worker is None:
            with torch.cuda.stream(self.side):
                self._side_part(j, s, factors, first_job, mark, hook)
            return
        ready = None
        if s == self.C - 1 and j - 1 >= first_job:
            ready = self._qd_ready[j - 1] = threading.Event()
        self._tasks.put(lambda: self._side_part(j, s, factors, first_job, mark, hook, ready))

    def join(self):
        """Make the current stream wait for the query side's work queued so far (and, with
        the query-side thread, wait until that thread has enqueued it)."""
        if self._worker is not None:
            self._tasks.join()
            if self._err is not None:
                err, self._err = self._err, None
                raise err
        if self.side is not None:
            torch.cuda.current_stream().wait_stream(self.side)

    def close(self):
        """Stop the query-side thread (after join())."""
        if self._worker is not None:
            self._tasks.put(None)
            self._worker.join()
            self._worker = None
