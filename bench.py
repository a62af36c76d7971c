#!/usr/bin/env python3
"""Throughput of the attribution hot path on GB300.

Workloads (--workload):

* llama3_8b_stack (default): a Llama-3-8B-shaped stack of 32 layers x 7 linears
  (q/o 4096x4096, k/v 4096->1024, gate/up 4096->14336, down 14336->4096), bf16,
  T = 1024 tokens, k_in = k_out = 64 (4096 features per linear, 917,504 per
  example), 8192 train examples streamed in chunks of 256, 256 queries,
  per-linear (F + lambda I)^-1 with lambda = 1e-2 x mean eigenvalue, top-100.
* large_model: one block of large-model layers (d_model 12288, ffn 49152, GQA
  k/v 12288->1536), bf16, T = 2048, k = 128 (16384 features per linear), 16384
  train examples in chunks of 512, 512 queries, A ~ Student-t(4), B ~ N(0,1e-4),
  lambda = 1e-2 x mean eigenvalue, top-100.
* llama1b_block: one Llama-style 1B block (q/k/v/o 2048x2048, gate/up
  2048->8192, down 8192->2048), T = 512, 4096 train / 64 query examples, k = 32,
  1% of tokens masked, every factor resident.

Stack workloads (paper_2609_38767_gb300.stream.StackJob): one step is one
chunk of train examples through the whole path -- the chunk's factored
projection through every linear and its Fisher sums, plus a 1/C share of the
previous job's query side (query projections, factorisation and
preconditioning, score) and of the job before's top-k, C = chunks per job. C
consecutive steps do exactly one job's work, so examples/s = chunk / step
time is whole-job throughput. Jobs run back to back; two jobs run untimed
first so that every share of the timed steps exists.

value: train examples attributed per second with the factors resident in HBM
(pools of examples larger than L2, so no flush is needed between steps; each
chunk of each layer reads its own window of the pool). e2e: the same steps
with the factors in pinned host memory through tda_project_host, the H2D
copies and the D2H read of the step's top-k rows inside the timed region.

--impl reference times the fp64 CPU oracle on a bounded sample of the same
workload on the host cores (the only other place this file runs the oracle).
"""
from __future__ import annotations

import argparse
import json
import math
import os
import statistics
import subprocess
import sys
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

LINEARS = [("q", 2048, 2048), ("k", 2048, 2048), ("v", 2048, 2048), ("o", 2048, 2048),
           ("gate", 2048, 8192), ("up", 2048, 8192), ("down", 8192, 2048)]
METRIC = "train examples attributed/sec (project+score)"

# DRAM traffic of the tensor-core projection kernel, from one ncu capture per k
# (dram__bytes_read.sum + dram__bytes_write.sum over the algorithmic bytes of the
# launch): k = 32, 608 examples of the 2048x2048 linear at T = 512; k = 64, 160
# examples of the 4096x4096 linear at T = 1024, whole examples per SM; k = 128, 32
# examples of the 12288 -> 1536 linear at T = 2048, balanced token-tile ranges
# (the ncu summaries under profiles/).
# Launches of other linears are scaled by their algorithmic bytes (every factor
# byte is read once, so traffic grows in proportion). Valid only for the kernel
# source it was measured on (the kernel file and its PTX helper header); any
# change makes the bench report null.
TRAFFIC_RATIO = {32: 1.0010593, 64: 1.0015892, 128: 1.0161220}
TRAFFIC_KERNEL_SHA256 = "c53a2d006d1a2c17ee9e12c8a801b33b575b313e63b0c1812a4e220a3a997072"


def projection_kernel_sha256():
    """sha256 of the projection kernel's code: k_project_tc.cu and tc_ptx.cuh with their
    // comments and blank lines removed (a comment edit does not change the kernel)."""
    import hashlib
    import re

    h = hashlib.sha256()
    for name in ("k_project_tc.cu", "tc_ptx.cuh"):
        with open(os.path.join(ROOT, "paper_2609_38767_gb300", "csrc", name)) as f:
            for line in f:
                code = re.sub(r"//.*$", "", line).rstrip()
                if code:
                    h.update(code.encode() + b"\n")
    return h.hexdigest()


def parse_args():
    p = argparse.ArgumentParser()
    p.add_argument("--gpus", type=int, default=1)
    p.add_argument("--steps", type=int, default=5)
    p.add_argument("--warmup", type=int, default=3)
    p.add_argument("--impl", default="ours", choices=["ours", "reference"])
    p.add_argument("--workload", default="llama3_8b_stack", choices=["llama3_8b_stack", "large_model", "llama1b_block"])
    p.add_argument("--n-train", type=int, default=4096)
    p.add_argument("--n-query", type=int, default=64)
    p.add_argument("--T", type=int, default=512)
    p.add_argument("--k", type=int, default=32)
    p.add_argument("--topk", type=int, default=100)
    p.add_argument("--no-precondition", action="store_true")
    p.add_argument("--curvature", default="fisher", choices=["fisher", "kfac", "ekfac"],
                   help="preconditioner: full empirical Fisher of the projected features, or K-FAC / EK-FAC "
                        "on the projected factors (damping 0.1 x mean eigenvalue)")
    p.add_argument("--overlap-sms", type=int, default=0,
                   help="Fisher query side on a second stream; the train projection leaves this many SMs free")
    p.add_argument("--train-streams", type=int, default=2,
                   help="stack workloads: streams the train projections of a chunk are spread over")
    p.add_argument("--query-side-stream", type=int, default=1,
                   help="stack workloads: 1 = the query side and top-k on a stream of their own beside the "
                        "next chunks' projections, 0 = in line after each chunk")
    p.add_argument("--query-priority", type=int, default=None,
                   help="priority of that stream (lower = higher; default: the workload's)")
    p.add_argument("--train-priority", type=int, default=None,
                   help="stack workloads: priority of the train projection streams (lower = higher)")
    p.add_argument("--bulk-priority", type=int, default=None,
                   help="stack workloads: run the query side's Fisher fit and query projections on a stream of "
                        "this priority (default: the workload's; none = on the query-side stream)")
    p.add_argument("--side-thread", type=int, default=-1,
                   help="stack workloads: 1 = a host thread of its own enqueues the query side (-1: the workload's)")
    p.add_argument("--query-streams", type=int, default=8,
                   help="streams the query projections of the linears are spread over (device-resident leg)")
    p.add_argument("--e2e-steps", type=int, default=2)
    p.add_argument("--no-e2e", action="store_true")
    p.add_argument("--no-cpu-baseline", action="store_true")
    p.add_argument("--pool", type=int, default=16, help="pinned host examples per linear for e2e")
    p.add_argument("--host-pool", type=int, default=None,
                   help="stack workloads: pinned host examples per linear shape for e2e (default: the workload's)")
    p.add_argument("--linears", default="q,k,v,o,gate,up,down",
                   help="subset of the block's linears (profiling of a smaller case)")
    p.add_argument("--project-only", action="store_true",
                   help="time only the train projection (kernel profiling; not the metric's step)")
    p.add_argument("--token-scores", action="store_true",
                   help="time token-level scores of the block (every train token against every preconditioned query)")
    p.add_argument("--masks", type=int, default=0,
                   help="time the random-mask reduction: ten disjoint masks of this many DW coordinates per linear")
    p.add_argument("--profile-project", default="",
                   help="stack workloads: time only the factored projection of this linear of a layer "
                        "(e.g. gate) over --profile-n examples, --steps launches (kernel profiling)")
    p.add_argument("--profile-precond", action="store_true",
                   help="stack workloads: time only one share's Fisher fit and factorisation with query solves "
                        "(one layer's linears, --profile-n train features) (kernel profiling)")
    p.add_argument("--profile-n", type=int, default=64)
    p.add_argument("--profile-linears", type=int, default=0,
                   help="--profile-precond: linears per call (0 = every linear of a layer)")
    p.add_argument("--sm-budget", type=int, default=None,
                   help="cap the persistent projection grid at this many CTAs (tda_set_sm_budget; 0 = every SM; "
                        "default: the workload's)")
    p.add_argument("--balance", type=int, default=-1,
                   help="stack workloads: 1 = balanced token-tile ranges in the train projections, 0 = whole "
                        "examples per SM, -1 = the workload's default")
    p.add_argument("--nvtx", action="store_true",
                   help="stack workloads: push an NVTX range 'timed' around the timed steps (for ncu --nvtx)")
    p.add_argument("--route-sweep", action="store_true",
                   help="route cost-model sweep on one 8192x8192 bf16 linear (chosen vs measured fastest route)")
    p.add_argument("--sweep-T", default="8,32,128,512,2048,8192")
    p.add_argument("--sweep-ops", default="project,similarity_projected,similarity_exact")
    p.add_argument("--sweep-routes", default="factored,materialize,gram")
    p.add_argument("--sweep-pool-gb", type=float, default=16.0, help="resident train factors per sweep point")
    p.add_argument("--sweep-d", type=int, default=8192, help="square linear d x d of the sweep")
    p.add_argument("--sweep-nq", type=int, default=128, help="queries of the sweep")
    a = p.parse_args()
    names = a.linears.split(",")
    global LINEARS
    LINEARS = [x for x in LINEARS if x[0] in names]
    return a


def workload(args):
    return {
        "workload": "llama1b_block_bf16",
        "linears": {n: [di, do] for n, di, do in LINEARS},
        "T": args.T, "n_train": args.n_train, "n_query": args.n_query,
        "k_in": args.k, "k_out": args.k, "features_per_example": len(LINEARS) * args.k * args.k,
        "factors": "A~N(0,1), B~N(0,1e-3), 1% tokens masked (seeded synthetic)",
        "method": ("GradDot" if args.no_precondition else
                   "(F+lambda I)^-1-preconditioned, lambda=1e-2*mean eig" if args.curvature == "fisher" else
                   f"{args.curvature.upper()} on projected factors, lambda=0.1*mean eig"),
        "topk": args.topk, "l2": "inputs larger than L2 (no flush)",
        "parallelism": "train examples sharded over the ranks (one GPU per rank)",
        **({"mode": "project-only (kernel profiling)"} if args.project_only else {}),
        **({"query_side": f"second stream beside the train projection, which leaves {args.overlap_sms} SMs free"}
           if getattr(args, "overlap_sms", 0) > 0 and not args.no_precondition and args.curvature == "fisher"
           and not args.project_only else {}),
    }


def _cpulist(text):
    cpus = set()
    for part in text.strip().split(","):
        if part:
            a, _, b = part.partition("-")
            cpus.update(range(int(a), int(b or a) + 1))
    return cpus


def bind_to_gpu_numa(index):
    """Pin this thread to the CPUs of the GPU's NUMA node (best effort).
    Returns (previous affinity or None, node or None)."""
    try:
        out = subprocess.run(["nvidia-smi", "--query-gpu=pci.bus_id", "--format=csv,noheader", "-i", str(index)],
                             capture_output=True, text=True, timeout=30).stdout.strip()
        dom, rest = out.split(":", 1)
        dev_path = "/sys/bus/pci/devices/%04x:%s/numa_node" % (int(dom, 16), rest.lower())
        with open(dev_path) as f:
            node = int(f.read().strip())
        if node < 0:
            return None, None
        with open("/sys/devices/system/node/node%d/cpulist" % node) as f:
            cpus = _cpulist(f.read()) & os.sched_getaffinity(0)
        if not cpus:
            return None, node
        saved = os.sched_getaffinity(0)
        os.sched_setaffinity(0, cpus)
        return saved, node
    except (OSError, ValueError, subprocess.SubprocessError):
        return None, None


# ---------------------------------------------------------------------------- clocks
class ClockSampler:
    FIELDS = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,clocks_event_reasons.hw_slowdown,"
              "clocks_event_reasons.hw_thermal_slowdown,clocks_event_reasons.sw_thermal_slowdown,"
              "clocks_event_reasons.sw_power_cap")

    def __init__(self, index):
        self.index = index
        self.proc = None

    def start(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.index), f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits",
                 "-lms", "100"], stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except OSError:
            self.proc = None

    def stop(self):
        if self.proc is None:
            return None
        self.proc.terminate()
        try:
            out, _ = self.proc.communicate(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
            out, _ = self.proc.communicate()
        rows = []
        for line in out.splitlines():
            parts = [x.strip() for x in line.split(",")]
            if len(parts) < 8:
                continue
            try:
                rows.append((float(parts[0]), float(parts[1]), parts[4:8]))
            except ValueError:
                continue
        if not rows:
            return None
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for _, _, flags in rows for i, f in enumerate(flags) if f.lower() == "active"})
        return {"sm_mhz": statistics.median(r[0] for r in rows), "sm_max_mhz": max(r[1] for r in rows),
                "reasons": reasons, "samples": len(rows)}


# ---------------------------------------------------------------------------- oracle (CPU)
def oracle_sample(args, n_s, n_q_s, factors_of):
    """Time the fp64 oracle on n_s train and n_q_s query examples of the block and
    extrapolate to the full workload's examples/s. factors_of(role, l, e0, n)
    returns float64 arrays (A, B) for n examples."""
    import numpy as np

    import oracle

    oracle.build()
    threads = os.cpu_count() or 1
    oracle.set_threads(threads)
    k, D = args.k, args.k * args.k
    t_train = t_query = t_fisher = t_factor = 0.0
    phis, qs = [], []
    for li, (_, di, do) in enumerate(LINEARS):
        A, B = factors_of("train", li, 0, n_s)
        t0 = time.perf_counter()
        phis.append(oracle.project(A, B, k, k, 0, li).reshape(n_s, D))
        t_train += time.perf_counter() - t0
        Aq, Bq = factors_of("query", li, 0, n_q_s)
        t0 = time.perf_counter()
        qs.append(oracle.project(Aq, Bq, k, k, 0, li).reshape(n_q_s, D))
        t_query += time.perf_counter() - t0
        if not args.no_precondition and args.curvature == "fisher":
            t0 = time.perf_counter()
            F = oracle.fisher(phis[-1])
            t_fisher += time.perf_counter() - t0
            t0 = time.perf_counter()
            qs[-1] = oracle.precondition(F, oracle.damping(F, 0.0, 1e-2), qs[-1])
            t_factor += time.perf_counter() - t0
        elif not args.no_precondition:
            # K-FAC / EK-FAC: covariances and EK-FAC eigenvalues per train example,
            # eigenbases once, the eigenbasis solve per query
            t0 = time.perf_counter()
            Ca, Cg = oracle.kfac_covariances(A, B, k, k, 0, li)
            t_fisher += time.perf_counter() - t0
            t0 = time.perf_counter()
            wa, Ua, _ = oracle.sym_eig(Ca)
            wg, Ug, _ = oracle.sym_eig(Cg)
            t_factor += time.perf_counter() - t0
            t0 = time.perf_counter()
            Lam = (oracle.ekfac_eigenvalues(phis[-1].reshape(n_s, k, k), Ua, Ug) if args.curvature == "ekfac"
                   else oracle.kfac_eigenvalues(wa, wg))
            t_fisher += time.perf_counter() - t0
            t0 = time.perf_counter()
            qs[-1] = oracle.kfac_precondition(Ua, Ug, Lam, oracle.kfac_damping(Lam, 0.0, 0.1), qs[-1])
            t_query += time.perf_counter() - t0
    t0 = time.perf_counter()
    S = oracle.score(np.concatenate(qs, 1), np.concatenate(phis, 1))
    oracle.topk(S, min(args.topk, n_s))
    t_score = time.perf_counter() - t0
    N, Nq = args.n_train, args.n_query
    total = (t_train + t_fisher + t_score * Nq / n_q_s) * N / n_s + t_query * Nq / n_q_s + t_factor
    fit = {"fisher": "Fisher/Cholesky", "kfac": "K-FAC covariances/eigenbases",
           "ekfac": "EK-FAC covariances/eigenbases/eigenvalues"}[args.curvature]
    sample = (f"{n_s} train + {n_q_s} query examples (fp64, {threads} threads) through all 7 linears, {fit}/score on them; "
              f"per-train-example parts scaled by {N}/{n_s}, query parts by {Nq}/{n_q_s}, factorisation once")
    return N / total, threads, sample, t_train + t_query + t_fisher + t_factor + t_score


def reference_main(args):
    """--impl reference: the oracle as it stands on the host cores, same config and metric."""
    import numpy as np

    from paper_2609_38767_gb300 import synth

    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return 0
    sb = math.sqrt(1e-3)

    cache = {}

    def factors_of(role, li, e0, n):
        # two generated examples per (role, linear), cycled to n: the oracle's work
        # does not depend on the values, and generation stays out of the timing
        key = (role, li)
        if key not in cache:
            di, do = LINEARS[li][1], LINEARS[li][2]
            off = synth.QUERY_STREAM_OFFSET if role == "query" else 0
            ms = 1000 if role == "query" else 0
            A = synth.factors(synth.SEED_A, li + off, 2, args.T, di, 1.0, 0, 0, "bf16", 0.01, mask_stream=ms)
            B = synth.factors(synth.SEED_B, li + off, 2, args.T, do, sb, 0, 0, "bf16", 0.01, mask_stream=ms)
            cache[key] = (synth.to_f64(A, "bf16"), synth.to_f64(B, "bf16"))
        A, B = cache[key]
        reps = (n + 1) // 2
        return np.tile(A, (reps, 1, 1))[:n], np.tile(B, (reps, 1, 1))[:n]

    threads = os.cpu_count() or 1
    n_s, n_q_s = max(2, threads), 2
    vals, secs = [], []
    sample = ""
    for i in range(args.warmup + args.steps):
        v, cores, sample, s = oracle_sample(args, n_s, n_q_s, factors_of)
        if i >= args.warmup:
            vals.append(v)
            secs.append(s)
    value = statistics.median(vals)
    line = {
        "impl": "reference", "metric": METRIC, "value": value, "unit": "examples/s", "n_gpus": args.gpus,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1e3 * statistics.median(secs),
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "config": workload(args),
        "cpu_baseline": {"value": value, "unit": "examples/s", "cores": cores, "kind": "oracle",
                         "sample": sample + "; ms_per_step is one sample's wall time"},
        "e2e": {"value": value, "unit": "examples/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)
    return 0


# ---------------------------------------------------------------------------- GPU arm
def route_sweep_main(args):
    """One 8192x8192 bf16 linear (--sweep-d), A, B ~ N(0,1), k = 64, 128 queries (--sweep-nq),
    N_train = 2^24 / T for each T:
    every route of every op is timed on the device and extrapolated to the full N_train by a
    two-point linear fit in the train count (t = a + b n); the route the Table 2 flop model
    picks and the one the calibrated model picks are reported beside the measured fastest."""
    import torch

    import paper_2609_38767_gb300 as tda
    from paper_2609_38767_gb300 import build as tbuild
    from paper_2609_38767_gb300 import synth

    tbuild.build()
    tda.load()
    dev = torch.device("cuda", 0)
    torch.cuda.set_device(dev)
    d, k, nq = args.sweep_d, 64, args.sweep_nq
    D = k * k
    cal_ws = torch.empty(tda.TDA_CALIBRATE_WS_BYTES, dtype=torch.uint8, device=dev)
    rates = tda.tda_route_calibrate(cal_ws, tda.TDA_CALIBRATE_WS_BYTES)
    del cal_ws
    names = {0: "factored", 1: "materialize", 2: "gram"}
    ops = [(tda.TDA_OP_PROJECT, "project", (0, 1)), (tda.TDA_OP_SIMILARITY_PROJECTED, "similarity_projected", (0, 1, 2)),
           (tda.TDA_OP_SIMILARITY_EXACT, "similarity_exact", (1, 2))]
    out = {"mode": "route-sweep", "linear": [d, d], "k": k, "n_query": nq, "dtype": "bf16",
           "calibrated_rates_tflops": dict(zip(("factored", "materialize_build", "gram_bf16", "gram_fp32",
                                                "dw_sign_projection", "dw_dots"), [r / 1e12 for r in rates[:6]])),
           "calibrated_bw_gbs": rates[6] / 1e9,
           "points": []}
    stream = torch.cuda.current_stream()
    for T in [int(x) for x in args.sweep_T.split(",")]:
        N = 2 ** 24 // T
        L = tda.LayerDesc(d, d, T, k, k, seed=0, layer=0)
        ex_bytes = T * 2 * d * 2
        P = max(1, min(N, int(args.sweep_pool_gb * 1e9 // ex_bytes)))
        A = torch.empty(P * T * d, dtype=torch.bfloat16, device=dev)
        B = torch.empty_like(A)
        Aq = torch.empty(nq * T * d, dtype=torch.bfloat16, device=dev)
        Bq = torch.empty_like(Aq)
        for x, seed, st in ((A, synth.SEED_A, 0), (B, synth.SEED_B, 0), (Aq, synth.SEED_A, 1000), (Bq, synth.SEED_B, 1000)):
            synth.fill_device(x, seed, st, x.numel() // (T * d), T, d, 1.0)
        phi = torch.empty(P * D, dtype=torch.float32, device=dev)
        S = torch.empty(nq * P, dtype=torch.float32, device=dev)

        def run(op, route, n_q, n_t, ws, wsb):
            done = 0
            while done < n_t:
                c = min(P, n_t - done)
                if op == tda.TDA_OP_PROJECT:
                    tda.tda_project(L, tda.TDA_BF16, A, B, c, phi, D, route, ws, wsb)
                elif op == tda.TDA_OP_SIMILARITY_PROJECTED:
                    tda.tda_similarity_projected(L, tda.TDA_BF16, Aq, Bq, n_q, A, B, c, S, c, 0.0, route, ws, wsb)
                else:
                    tda.tda_similarity_exact(L, tda.TDA_BF16, Aq, Bq, n_q, A, B, c, S, c, 0.0, route, ws, wsb)
                done += c

        def timed(op, route, n_q, n_t, ws, wsb):
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record(stream)
            run(op, route, n_q, n_t, ws, wsb)
            e1.record(stream)
            e1.synchronize()
            return e0.elapsed_time(e1) * 1e-3

        point = {"T": T, "n_train": N, "pool_examples": P, "ops": {}}
        for op, opname, routes in ops:
            if opname not in args.sweep_ops.split(","):
                continue
            routes = tuple(r for r in routes if names[r] in args.sweep_routes.split(","))
            rec = {"flop_model_choice": names[tda.tda_route(L, op, nq, N, tda.TDA_BF16)[0]]}
            tda.tda_route_set_model(1)
            ch, est = tda.tda_route(L, op, nq, N, tda.TDA_BF16)
            tda.tda_route_set_model(0)
            rec["calibrated_choice"] = names[ch]
            rec["calibrated_estimate_s"] = {names[r]: est[r] for r in routes}
            meas = {}
            for r in routes:
                n_q = nq
                # start with enough train examples to fill the GPU (the fit below is in the train count)
                n1 = min(P, 8)
                wsb = max(tda.tda_workspace_size(op, L, tda.TDA_BF16, n_q, P, r), 256)
                if op == tda.TDA_OP_SIMILARITY_EXACT and r == 1:
                    # materialised train gradients go through in chunks, each chunk re-reading the
                    # queries' DW: time whole chunks (one and two per call) so that cost lands in the slope
                    chunk = max(1, min(128, P // 2))
                    wsb = tda.tda_workspace_size(op, L, tda.TDA_BF16, n_q + chunk - 1, P, r)
                    n1 = chunk
                if op == tda.TDA_OP_SIMILARITY_PROJECTED:
                    wsb = max(wsb, min(2 << 30, tda.tda_workspace_size(op, L, tda.TDA_BF16, n_q, P, r) * 16))
                ws = torch.empty(wsb, dtype=torch.uint8, device=dev)
                timed(op, r, n_q, n1, ws, wsb)  # warm-up
                t1 = timed(op, r, n_q, n1, ws, wsb)
                while t1 < 0.05 and n1 < N and not (op == tda.TDA_OP_SIMILARITY_EXACT and r == 1):
                    n1 = min(N, n1 * max(2, int(0.1 / max(t1, 1e-6))))
                    t1 = timed(op, r, n_q, n1, ws, wsb)
                if 2 * n1 <= N:
                    t2 = timed(op, r, n_q, 2 * n1, ws, wsb)
                    b = max((t2 - t1) / n1, 0.0)
                    a = max(t1 - b * n1, 0.0)
                else:
                    a, b = 0.0, t1 / n1
                full = (a + b * N) * (nq / n_q)
                meas[names[r]] = {"seconds": full, "timed_train_examples": [n1, 2 * n1 if 2 * n1 <= N else n1],
                                  "timed_queries": n_q, "extrapolated": n1 < N or n_q < nq}
                del ws
                torch.cuda.synchronize()
            fastest = min(meas, key=lambda x: meas[x]["seconds"])
            rec["measured"] = meas
            rec["measured_fastest"] = fastest
            for key, choice in (("calibrated_over_fastest", rec["calibrated_choice"]),
                                ("flop_model_over_fastest", rec["flop_model_choice"])):
                rec[key] = meas[choice]["seconds"] / meas[fastest]["seconds"] if choice in meas else None
            point["ops"][opname] = rec
        tda.tda_device_status()
        out["points"].append(point)
        print(json.dumps(point), file=sys.stderr, flush=True)
        del A, B, Aq, Bq, phi, S
        torch.cuda.empty_cache()
    print(json.dumps(out))


def reuse_main(args):
    """Two reuses of the block's factors, timed like the main step: token-level scores
    (every train token against every preconditioned query, summed over the linears) or the
    random-mask reduction (ten disjoint masks of --masks coordinates per linear, gathered
    for train and query examples, then one score GEMM over the concatenated masks)."""
    import numpy as np
    import torch

    import paper_2609_38767_gb300 as tda
    from paper_2609_38767_gb300 import build as tbuild
    from paper_2609_38767_gb300 import synth
    from paper_2609_38767_gb300.block import BlockPipeline

    tbuild.build()
    tda.load()
    dev = torch.device("cuda", 0)
    torch.cuda.set_device(dev)
    stream = torch.cuda.current_stream()
    T, N, Nq, k = args.T, args.n_train, args.n_query, args.k
    D, nl = k * k, len(LINEARS)
    DT = D * nl
    sb = math.sqrt(1e-3)
    At, Bt, Aq, Bq = [], [], [], []
    for li, (_, di, do) in enumerate(LINEARS):
        for store, n, role, seed, d, sg in ((At, N, 0, synth.SEED_A, di, 1.0), (Aq, Nq, 1, synth.SEED_A, di, 1.0),
                                            (Bt, N, 0, synth.SEED_B, do, sb), (Bq, Nq, 1, synth.SEED_B, do, sb)):
            x = torch.empty((n, T, d), dtype=torch.bfloat16, device=dev)
            synth.fill_device(x, seed, li + (synth.QUERY_STREAM_OFFSET if role else 0), n, T, d, sg, mask_p=0.01,
                              mask_stream=1000 if role else 0)
            store.append(x)
    pipe = BlockPipeline([(di, do) for _, di, do in LINEARS], T, k, N, Nq, topk=args.topk, lambda_rel=1e-2,
                         device=dev)
    layers = pipe.layers

    def proj(role, li, L, route, phi, ld):
        X, Y, n = (At[li], Bt[li], N) if role == "train" else (Aq[li], Bq[li], Nq)
        tda.tda_project(L, tda.TDA_BF16, X, Y, n, phi, ld, route)

    pipe.run(lambda *a: proj("train", *a), lambda *a: proj("query", *a))  # preconditioned queries, untimed
    torch.cuda.synchronize()
    if args.token_scores:
        out = torch.empty((Nq, N * T), dtype=torch.float32, device=dev)
        # 1024 examples per chunk, plus room for the query matrices' hi/lo halves (tensor-core contraction)
        wsb = max(tda.tda_token_scores_workspace_size(L) for L in layers) * 1024 + (4 << 20)
        ws = torch.empty(wsb, dtype=torch.uint8, device=dev)

        def step():
            for li, L in enumerate(layers):
                tda.tda_token_scores(L, tda.TDA_BF16, At[li], Bt[li], N, pipe.Qh[:, li * D:], Nq, DT, out, N * T,
                                     0.0 if li == 0 else 1.0, ws, wsb)

        flops = sum(N * 2.0 * T * (L.d_in + L.d_out) * k + 2.0 * Nq * N * T * D for L in layers)
        # the step reads every factor once (projection, HBM-bound) and then contracts the projected
        # factors on the tensor cores; the roofline is the whole step against reading the factors
        fbytes = sum(2.0 * N * T * (L.d_in + L.d_out) for L in layers)
        mode = {"mode": "token-level scores", "n_query": Nq, "outputs_per_step": Nq * N * T,
                "contraction_tflop_per_step": 2.0 * Nq * N * T * D * nl / 1e12}
        roof_kernel, roof_bound = "factor projection (tcgen05) + token contraction (tcgen05, 3xTF32), whole step", "hbm"
    else:
        K = args.masks
        rng = np.random.default_rng(2026)
        coords = []
        for L in layers:
            flat = rng.choice(L.d_in * L.d_out, size=10 * K, replace=False)
            coords.append((torch.from_numpy((flat // L.d_in).astype(np.int32)).to(dev),
                           torch.from_numpy((flat % L.d_in).astype(np.int32)).to(dev)))
        nc = 10 * K
        Gt = torch.empty((N, nl * nc), dtype=torch.float32, device=dev)
        Gq = torch.empty((Nq, nl * nc), dtype=torch.float32, device=dev)

        def step():
            for li, L in enumerate(layers):
                r, c = coords[li]
                tda.tda_mask_gather(L, tda.TDA_BF16, At[li], Bt[li], N, r, c, nc, Gt[:, li * nc:], nl * nc)
                tda.tda_mask_gather(L, tda.TDA_BF16, Aq[li], Bq[li], Nq, r, c, nc, Gq[:, li * nc:], nl * nc)
            tda.tda_score(Gq, tda.TDA_F32, Nq, nl * nc, Gt, N, nl * nc, nl * nc, pipe.S, N, 0.0)
            tda.tda_topk(pipe.S, Nq, N, N, args.topk, pipe.idx, pipe.val)

        flops = sum(2.0 * (N + Nq) * T * nc for L in layers) + 2.0 * Nq * N * nl * nc
        mode = {"mode": "random-mask reduction", "masks_per_linear": 10, "coordinates_per_mask": K}
        roof_kernel, roof_bound = "mask gather + score", "alu"
    for _ in range(max(args.warmup, 1)):
        step()
    tda.tda_device_status()
    torch.cuda.synchronize()
    clocks = ClockSampler(0)
    clocks.start()
    time.sleep(0.3)
    l0 = tda.tda_launch_count()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for _ in range(args.steps):
        step()
    e1.record(stream)
    torch.cuda.synchronize()
    launches = tda.tda_launch_count() - l0
    ck = clocks.stop()
    tda.tda_device_status()
    ms = e0.elapsed_time(e1) / args.steps
    peaks = {}
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            peaks = json.load(f)
    except OSError:
        pass
    alu = 152 * 128 * 2 * float(peaks.get("sm_max_mhz", 2070.0)) * 1e6 / 1e12
    rate = flops / (ms * 1e-3) / 1e12
    if roof_bound == "hbm":
        hbm = float(peaks.get("hbm_gbs", 6794.1))
        roof = {"bound": "hbm", "kernel": roof_kernel, "achieved": fbytes / (ms * 1e-3) / 1e9, "peak": hbm,
                "unit": "GB/s", "frac": fbytes / (ms * 1e-3) / 1e9 / hbm, "traffic": None,
                "peak_source": "MEASURED_PEAKS.json hbm_gbs (copy)"}
    else:
        roof = {"bound": roof_bound, "kernel": roof_kernel, "achieved": rate, "peak": alu, "unit": "TFLOP/s",
                "frac": rate / alu, "traffic": None,
                "peak_source": "fp32 SIMT peak derived from 152 SMs x 128 lanes x 2 x max clock"}
    print(json.dumps({
        "metric": METRIC, "value": N / (ms * 1e-3), "unit": "examples/s", "n_gpus": 1, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": ms, "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
        "dtype": "bf16", "data": "synthetic", "config": {**workload(args), **mode},
        "roofline": roof,
        "cpu_baseline": None, "e2e": None, "gpu_launches": launches, "clocks": ck}))


# ---------------------------------------------------------------------------- streamed stacks
STACKS = {
    "llama3_8b_stack": {
        "layer": [("q", 4096, 4096), ("k", 4096, 1024), ("v", 4096, 1024), ("o", 4096, 4096),
                  ("gate", 4096, 14336), ("up", 4096, 14336), ("down", 14336, 4096)],
        "n_layers": 32, "T": 1024, "k": 64, "n_train": 8192, "chunk": 256, "n_query": 256,
        "dist_a": 0, "sigma_b": math.sqrt(1e-3), "lambda_rel": 1e-2,
        "train_pool": 512, "query_pool": 256, "host_pool": 4, "balance": False, "query_priority": 0, "sm_budget": 0,
        "factors": "A~N(0,1), B~N(0,1e-3) (seeded synthetic)",
    },
    "large_model": {
        "layer": [("q", 12288, 12288), ("k", 12288, 1536), ("v", 12288, 1536), ("o", 12288, 12288),
                  ("gate", 12288, 49152), ("up", 12288, 49152), ("down", 49152, 12288)],
        "n_layers": 1, "T": 2048, "k": 128, "n_train": 16384, "chunk": 512, "n_query": 512,
        "dist_a": 1, "sigma_b": 0.01, "lambda_rel": 1e-2,
        "train_pool": 128, "query_pool": 64, "host_pool": 16, "balance": True, "query_priority": -1, "sm_budget": 128,
        "factors": "A~Student-t(4), B~N(0,1e-4) (seeded synthetic)",
    },
}


def stack_config(args, spec):
    lin = spec["layer"]
    nlin = len(lin) * spec["n_layers"]
    D = spec["k"] ** 2
    return {
        "workload": args.workload,
        "linears_per_layer": {n: [di, do] for n, di, do in lin}, "layers": spec["n_layers"],
        "T": spec["T"], "n_train": spec["n_train"], "chunk": spec["chunk"], "n_query": spec["n_query"],
        "k_in": spec["k"], "k_out": spec["k"], "features_per_example": nlin * D,
        "factors": spec["factors"],
        "method": f"(F+lambda I)^-1-preconditioned per linear, lambda={spec['lambda_rel']:g}*mean eig",
        "topk": args.topk,
        "step": (f"one chunk of {spec['chunk']} train examples projected through all {nlin} linears + "
                 f"1/{spec['n_train'] // spec['chunk']} of the previous job's query side (Fisher fit over the "
                 "job's resident features, query projection, factorisation + preconditioning, score) and of the "
                 "job before's top-k"),
        "resident_pools": (f"{spec['train_pool']} train / {spec['query_pool']} query examples per linear shape in "
                           "HBM; each (chunk, layer) reads its own window of the train pool"),
        "l2": "inputs larger than L2 (no flush)",
        "parallelism": ("one GPU" if int(os.environ.get("WORLD_SIZE", "1")) == 1 else
                        f"replicas: an independent job on each of {os.environ.get('WORLD_SIZE')} GPUs"),
        "routes": "factored (every linear)",
        "train_schedule": ("balanced token-tile ranges per launch"
                           if (spec["balance"] if args.balance < 0 else bool(args.balance))
                           else "whole examples per SM") + f", {args.train_streams} train streams"
                          + (lambda b: f", projection grids capped at {b} CTAs" if b else "")(
                              spec["sm_budget"] if args.sm_budget is None else args.sm_budget),
    }


def stack_oracle_sample(spec, factors_of):
    """Time the fp64 oracle on a bounded sample of a stack job and extrapolate to the job's
    examples/s: n_s train and 2 query examples through the first two linears of one layer (q
    and k; the oracle's projection time is proportional to T (d_in + d_out) per example, so
    it is scaled to the layer's seven linears by that sum), the Fisher of one linear over the
    n_s train features, the damped inverse (D x D Cholesky) applied to the queries, and their
    scores. factors_of(role, li, n) returns float64 (A, B)."""
    import numpy as np

    import oracle

    oracle.build()
    threads = os.cpu_count() or 1
    oracle.set_threads(threads)
    n_s, nq_s, k, D = max(2, threads), 2, spec["k"], spec["k"] ** 2
    sampled = (0, 1)
    width = lambda li: spec["layer"][li][1] + spec["layer"][li][2]
    scale = sum(width(li) for li in range(len(spec["layer"]))) / sum(width(li) for li in sampled)
    t_proj = t_qproj = 0.0
    phis, qs = [], []
    for li in sampled:
        A, B = factors_of("train", li, n_s)
        t0 = time.perf_counter()
        phis.append(oracle.project(A, B, k, k, 0, li).reshape(n_s, D))
        t_proj += time.perf_counter() - t0
        Aq, Bq = factors_of("query", li, nq_s)
        t0 = time.perf_counter()
        qs.append(oracle.project(Aq, Bq, k, k, 0, li).reshape(nq_s, D))
        t_qproj += time.perf_counter() - t0
    t0 = time.perf_counter()
    F = oracle.fisher(phis[0])
    t_fit = time.perf_counter() - t0
    t0 = time.perf_counter()
    qh = oracle.precondition(F, oracle.damping(F, 0.0, spec["lambda_rel"]), qs[0])
    t_fact = time.perf_counter() - t0
    t0 = time.perf_counter()
    S = oracle.score(qh, phis[0])
    oracle.topk(S, 1)
    t_score = time.perf_counter() - t0
    N, Nq, L = spec["n_train"], spec["n_query"], spec["n_layers"]
    nlin = L * len(spec["layer"])
    total = (t_proj * scale * L * N / n_s + t_qproj * scale * L * Nq / nq_s + t_fit * nlin * N / n_s
             + t_fact * nlin + t_score * nlin * (N / n_s) * (Nq / nq_s))
    sample = (f"{n_s} train + {nq_s} query examples (fp64, {threads} threads) through the q and k linears of one "
              f"layer, Fisher of one linear over them, D x D Cholesky + solves, scores; projection scaled by "
              f"{scale:.2f} (the layer's sum of d_in + d_out over q's and k's) x {L} layers x {N}/{n_s} (queries "
              f"{Nq}/{nq_s}), Fisher by {nlin} linears x {N}/{n_s}, factorisation by {nlin} linears, score by "
              f"{nlin} x {N}/{n_s} x {Nq}/{nq_s}")
    wall = t_proj + t_qproj + t_fit + t_fact + t_score
    return N / total, threads, sample, wall


def stack_factors_host(spec, li, role, n):
    """float64 factors of n examples of linear li of the layer (for the oracle sample)."""
    from paper_2609_38767_gb300 import synth

    _, di, do = spec["layer"][li]
    off = synth.QUERY_STREAM_OFFSET if role == "query" else 0
    A = synth.factors(synth.SEED_A, li + off, n, spec["T"], di, 1.0, spec["dist_a"], 0, "bf16")
    B = synth.factors(synth.SEED_B, li + off, n, spec["T"], do, spec["sigma_b"], 0, 0, "bf16")
    return synth.to_f64(A, "bf16"), synth.to_f64(B, "bf16")


def stack_reference_main(args, spec):
    if int(os.environ.get("RANK", "0")) != 0:
        return 0
    cache = {}

    def factors_of(role, li, n):
        key = (role, li, n)
        if key not in cache:
            cache[key] = stack_factors_host(spec, li, role, n)
        return cache[key]

    factors_of("train", 0, max(2, os.cpu_count() or 1))  # generation stays out of the timing
    vals, walls = [], []
    sample, cores = "", 1
    for i in range(args.warmup + args.steps):
        v, cores, sample, wall = stack_oracle_sample(spec, factors_of)
        if i >= args.warmup:
            vals.append(v)
            walls.append(wall)
    value = statistics.median(vals)
    line = {
        "impl": "reference", "metric": METRIC, "value": value, "unit": "examples/s", "n_gpus": args.gpus,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1e3 * statistics.median(walls),
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "config": stack_config(args, spec),
        "cpu_baseline": {"value": value, "unit": "examples/s", "cores": cores, "kind": "oracle",
                         "sample": sample + "; ms_per_step is one sample's wall time"},
        "e2e": {"value": value, "unit": "examples/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)
    return 0


def stack_profile_main(args, spec):
    """Small cases of the stack workloads' dominant kernels for ncu: one linear's factored
    projection, or one share's Fisher fit + factorisation with the query solves."""
    import torch

    import paper_2609_38767_gb300 as tda
    from paper_2609_38767_gb300 import build as tbuild
    from paper_2609_38767_gb300 import synth

    tbuild.build()
    tda.load()
    tda.tda_set_sm_budget(args.sm_budget or 0)
    dev = torch.device("cuda", 0)
    torch.cuda.set_device(dev)
    stream = torch.cuda.current_stream()
    T, k, n = spec["T"], spec["k"], args.profile_n
    D = k * k
    ev0, ev1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    if args.profile_project:
        li = [x[0] for x in spec["layer"]].index(args.profile_project)
        _, di, do = spec["layer"][li]
        A = torch.empty((n, T, di), dtype=torch.bfloat16, device=dev)
        B = torch.empty((n, T, do), dtype=torch.bfloat16, device=dev)
        synth.fill_device(A, synth.SEED_A, li, n, T, di, 1.0, spec["dist_a"])
        synth.fill_device(B, synth.SEED_B, li, n, T, do, spec["sigma_b"])
        L = tda.LayerDesc(di, do, T, k, k, seed=0, layer=li)
        assert tda.tda_project_engine(L, tda.TDA_BF16, A, B) == 1
        wsb = tda.tda_workspace_size(tda.TDA_OP_PROJECT, L, tda.TDA_BF16, n, 0, tda.TDA_ROUTE_FACTORED)
        if not (spec["balance"] if args.balance < 0 else bool(args.balance)):
            wsb = 2 * k * (di + do) if k == 128 else 0  # sign tables only: whole examples per SM
        ws = torch.empty(max(wsb, 256), dtype=torch.uint8, device=dev)
        phi = torch.empty((n, D), device=dev)
        run = lambda: tda.tda_project(L, tda.TDA_BF16, A, B, n, phi, D, tda.TDA_ROUTE_FACTORED, ws, wsb)
        work = ("GB/s", n * (T * (di + do) * 2 + 4 * D) / 1e9)
        what = {"kernel": "factored projection", "linear": [di, do], "n": n, "T": T, "k": k,
                "sign_tables": k == 128 and bool(wsb), "balanced": wsb > 2 * k * (di + do) * (k == 128)}
    else:
        nl = args.profile_linears or len(spec["layer"])
        per = tda.tda_precondition_state_bytes(D, tda.TDA_F32)
        st = torch.empty(nl * per, dtype=torch.uint8, device=dev)
        phi = torch.empty(n * nl * D, dtype=torch.float32, device=dev)
        synth.fill_device(phi, 5, 0, n, 1, nl * D, 1.0)
        q = torch.empty(spec["n_query"] * nl * D, dtype=torch.float32, device=dev)
        synth.fill_device(q, 6, 0, spec["n_query"], 1, nl * D, 1.0)
        qh = torch.empty_like(q)
        Nq = spec["n_query"]

        def run():
            tda.tda_precondition(tda.TDA_PC_RESET, nl, D, tda.TDA_F32, st)
            tda.tda_precondition(tda.TDA_PC_FIT_ACCUM, nl, D, tda.TDA_F32, st, phi=phi, n=n, ld_phi=nl * D)
            tda.tda_precondition(tda.TDA_PC_FACTOR_APPLY, nl, D, tda.TDA_F32, st, n_total=n,
                                 lambda_rel_mean_eig=spec["lambda_rel"], q=q, n_q=Nq, ld_q=nl * D, qhat=qh,
                                 ld_qhat=nl * D)
        work = ("TFLOP/s", nl * (n * D * (D + 1) + D ** 3 / 3 + 2 * D * D * Nq) / 1e12)
        what = {"kernel": "Fisher fit + factorisation + query solves", "linears": nl, "D": D, "n_train": n,
                "n_query": Nq}
    for _ in range(max(args.warmup, 1)):
        run()
    torch.cuda.synchronize()
    ev0.record(stream)
    for _ in range(args.steps):
        run()
    ev1.record(stream)
    torch.cuda.synchronize()
    tda.tda_device_status()
    ms = ev0.elapsed_time(ev1) / args.steps
    print(json.dumps({"mode": "profile", **what, "sm_budget": args.sm_budget or 0, "ms_per_call": ms,
                      "rate": work[1] / (ms * 1e-3), "unit": work[0]}))
    return 0


def stack_main(args, spec):
    import numpy as np
    import torch

    import paper_2609_38767_gb300 as tda
    from paper_2609_38767_gb300 import build as tbuild
    from paper_2609_38767_gb300 import synth
    from paper_2609_38767_gb300.stream import StackJob

    # Under torchrun every rank runs an independent replica of the job on its own GPU (the
    # method runs on one GPU; replicas share nothing): barrier and max over ranks around the
    # timed region, value = the replicas' examples over that time.
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    dev = torch.device("cuda", local)
    torch.cuda.set_device(dev)
    dist = None
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", device_id=dev)
    if rank == 0:
        tbuild.build()
    if dist:
        dist.barrier()
    tda.load()
    sm_budget = spec["sm_budget"] if args.sm_budget is None else args.sm_budget
    tda.tda_set_sm_budget(sm_budget)

    def max_over_ranks(x):
        if not dist:
            return x
        t = torch.tensor([x], dtype=torch.float64, device=dev)
        dist.all_reduce(t, op=dist.ReduceOp.MAX)
        return float(t.item())
    stream = torch.cuda.current_stream()
    lin, L = spec["layer"], spec["n_layers"]
    T, k, N, chunk, Nq = spec["T"], spec["k"], spec["n_train"], spec["chunk"], spec["n_query"]
    D = k * k
    C = N // chunk
    nshape = len(lin)
    linears = [(di, do) for _ in range(L) for _, di, do in lin]
    nlin = len(linears)
    steps = args.steps
    if (nlin % C or Nq % C) and steps % C:
        steps = (steps + C - 1) // C * C  # unequal shares per step: time whole jobs
    Pt, Pq = spec["train_pool"], spec["query_pool"]

    # ---- resident pools (untimed): per linear shape, Pt train and Pq query examples
    pools = []
    for si, (_, di, do) in enumerate(lin):
        ent = []
        for n, off, seed, d, sg, dist in ((Pt, 0, synth.SEED_A, di, 1.0, spec["dist_a"]),
                                          (Pt, 0, synth.SEED_B, do, spec["sigma_b"], 0),
                                          (Pq, synth.QUERY_STREAM_OFFSET, synth.SEED_A, di, 1.0, spec["dist_a"]),
                                          (Pq, synth.QUERY_STREAM_OFFSET, synth.SEED_B, do, spec["sigma_b"], 0)):
            x = torch.empty((n, T, d), dtype=torch.bfloat16, device=dev)
            synth.fill_device(x, seed, si + off, n, T, d, sg, dist, mask_stream=1000 if off else 0)
            ent.append(x)
        pools.append(ent)

    def window(li, j, s):
        """First pool row of chunk s of job j for linear li (a pseudo-random window per chunk and layer)."""
        layer = li // nshape
        span = Pt - chunk + 1 if Pt >= chunk else Pt
        return (131 * s + 37 * layer + 71 * j) % span

    def dev_factors(role, li, j, s):
        A, B, Aq, Bq = pools[li % nshape]
        if role == "train":
            if Pt >= chunk:
                o = window(li, j, s)
                return [(A[o:o + chunk], B[o:o + chunk], 0, chunk)]
            return [(A[:min(Pt, chunk - r)], B[:min(Pt, chunk - r)], r, min(Pt, chunk - r)) for r in range(0, chunk, Pt)]
        return [(Aq[:min(Pq, Nq - r)], Bq[:min(Pq, Nq - r)], r, min(Pq, Nq - r)) for r in range(0, Nq, Pq)]

    balance = spec["balance"] if args.balance < 0 else bool(args.balance)
    job = StackJob(linears, T, k, N, chunk, Nq, topk=args.topk, lambda_rel=spec["lambda_rel"], device=dev,
                   train_streams=args.train_streams, query_stream=bool(args.query_side_stream),
                   query_priority=spec["query_priority"] if args.query_priority is None else args.query_priority,
                   balance=balance,
                   train_priority=spec.get("train_priority", 0) if args.train_priority is None else args.train_priority,
                   bulk_priority=spec.get("bulk_priority") if args.bulk_priority is None else args.bulk_priority,
                   side_thread=spec.get("side_thread", False) if args.side_thread < 0 else bool(args.side_thread))
    for si in range(nshape):  # every linear shape runs on the tensor-core projection kernel
        assert tda.tda_project_engine(job.layers[si], tda.TDA_BF16, pools[si][0], pools[si][1]) == 1
    state = {"j": 0, "s": 0}

    def advance(factors, mark=None, hook=None):
        job.step(state["j"], state["s"], factors, mark=mark, hook=hook)
        state["s"] += 1
        if state["s"] == C:
            state["s"], state["j"] = 0, state["j"] + 1

    for _ in range(2 * C):  # two jobs: every share of the following steps exists
        advance(dev_factors)
    for _ in range(args.warmup):
        advance(dev_factors)
    job.join()
    tda.tda_device_status()
    torch.cuda.synchronize()

    ev, phase_ev, open_ev = [], [], {}
    # timing events created before the timed region (creating hundreds per step would add host
    # time to every step): two per train launch and about ten phase marks per step
    pool = [torch.cuda.Event(enable_timing=True) for _ in range(steps * (2 * nlin * (1 + max(1, chunk // Pt)) + 16))]

    def new_event():
        return pool.pop() if pool else torch.cuda.Event(enable_timing=True)

    def mark(name):
        st = torch.cuda.current_stream()  # phases are timed on the stream they run on
        e = new_event()
        e.record(st)
        phase_ev.append((name, e, st.cuda_stream))

    def hook(role, li, when, n):
        if role != "train":
            return
        e = new_event()
        e.record(torch.cuda.current_stream())
        if when == "begin":
            open_ev[li] = e
        else:
            di, do = linears[li]
            ev.append((open_ev.pop(li), e, n * (T * (di + do) * 2 + 4 * D)))

    clocks = ClockSampler(local)
    clocks.start()
    time.sleep(0.3)
    l0 = tda.tda_launch_count()
    t0, t1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    if dist:
        dist.barrier()
    torch.cuda.synchronize()
    if args.nvtx:
        torch.cuda.nvtx.range_push("timed")
    t0.record(stream)
    h0 = time.perf_counter()
    for _ in range(steps):
        advance(dev_factors, mark, hook)
    host_ms = (time.perf_counter() - h0) * 1e3 / steps  # host time to enqueue a step
    job.join()  # the query side queued in the timed steps is inside the timed region
    t1.record(stream)
    if args.nvtx:
        torch.cuda.nvtx.range_pop()
    torch.cuda.synchronize()
    if dist:
        dist.barrier()
    launches = tda.tda_launch_count() - l0
    ck = clocks.stop()
    tda.tda_device_status()
    ms = max_over_ranks(t0.elapsed_time(t1) / steps)
    value = world * chunk / (ms * 1e-3)

    peaks = {}
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            peaks = json.load(f)
    except OSError:
        pass
    hbm = float(peaks.get("hbm_gbs", 6800.0))
    tf32x3 = float(peaks.get("bf16_tflops_sustained", 1700.0)) * 0.5 / 3.0
    # the train projections of a step overlap across streams: the kernel's rate is its phase's
    # algorithmic bytes over the phase's time (events on the launching stream around the fork
    # and join of the projection streams)
    proj_bytes = sum(x for _, _, x in ev)
    seqs = {}
    for name, e, sid in phase_ev:
        seqs.setdefault(sid, []).append((name, e))
    ph = {}
    for seq in seqs.values():
        for (name, a), (_, b) in zip(seq, seq[1:]):
            if name is not None:
                ph[name] = ph.get(name, 0.0) + a.elapsed_time(b) / steps
    ph_train = ph.get("project_train", 0.0) * steps
    achieved = proj_bytes / (ph_train * 1e-3) / 1e9
    per_launch = proj_bytes / max(len(ev), 1)
    roofline = {"bound": "hbm", "kernel": f"factored projection (train, k = {k}, tcgen05)", "achieved": achieved,
                "peak": hbm, "unit": "GB/s", "frac": achieved / hbm,
                "traffic": None, "algorithmic_bytes_per_launch": per_launch, "launches_timed": len(ev),
                "timing": (f"train projection phase of each step ({len(ev) // steps} launches over "
                           f"{args.train_streams} stream(s)), CUDA events"),
                "peak_source": "MEASURED_PEAKS.json hbm_gbs" if peaks else "fallback 6.8 TB/s",
                "share_of_step": ph_train / (ms * steps)}
    if k in TRAFFIC_RATIO and projection_kernel_sha256() == TRAFFIC_KERNEL_SHA256:
        roofline["traffic"] = TRAFFIC_RATIO[k] * per_launch
        roofline["traffic_source"] = f"ncu dram bytes / algorithmic bytes of one k = {k} launch, scaled per launch"
    Dn = float(D)
    per_job_lin = {
        "project_train": ("hbm", sum(N * (T * (di + do) * 2 + 4 * D) for di, do in linears), hbm, "GB/s"),
        "fisher_fit": ("tensor", nlin * N * Dn * (Dn + 1), tf32x3, "TFLOP/s"),
        "project_query": ("hbm", sum(Nq * (T * (di + do) * 2 + 4 * D) for di, do in linears), hbm, "GB/s"),
        # Cholesky D^3/3 flops, the two triangular solves 2 D^2 flops per query
        "factor_apply": ("tensor", nlin * (Dn ** 3 / 3 + 2 * Dn * Dn * Nq), tf32x3, "TFLOP/s"),
        "score": ("tensor", 2.0 * Nq * N * D * nlin, tf32x3, "TFLOP/s"),
        "topk": ("latency", 4.0 * Nq * N, hbm, "GB/s"),
    }
    phases = {}
    side = bool(args.query_side_stream)
    for name, ms_ in ph.items():
        bound, work, peak, unit = per_job_lin[name]
        rate = work / C / (ms_ * 1e-3) / (1e9 if unit == "GB/s" else 1e12)
        phases[name] = {"ms": ms_, "bound": bound, "achieved": rate, "peak": peak, "unit": unit, "frac": rate / peak}
        if side and name != "project_train":
            # wall time on the query-side stream, beside the train projections that hold most SMs
            phases[name]["stream"] = "query side, overlapped"

    # ---- e2e: the same steps with the factors in pinned host memory
    e2e = None
    if not args.no_e2e:
        saved_aff, numa = bind_to_gpu_numa(local)
        Ph = spec["host_pool"] if args.host_pool is None else args.host_pool
        hpools = []
        for si in range(nshape):
            A, B, Aq, Bq = pools[si]
            hp = []
            for x in (A, B, Aq, Bq):
                h = torch.empty((Ph,) + tuple(x.shape[1:]), dtype=torch.bfloat16).pin_memory()
                h.copy_(x[:Ph])
                hp.append(h)
            hpools.append(hp)
        wsb = 2 * Ph * T * max(di + do for _, di, do in lin) * 2
        # room for the projection's own workspace beside each staging half (balanced tile ranges)
        pws = max(tda.tda_workspace_size(tda.TDA_OP_PROJECT, Lr, tda.TDA_BF16, 1, 0, tda.TDA_ROUTE_FACTORED)
                  for Lr in job.layers[:nshape])
        wsb += 2 * ((pws + 255) // 256 * 256)
        job.host_ws_bytes = wsb
        job.host_ws = torch.empty(wsb, dtype=torch.uint8, device=dev)

        def host_factors(role, li, j, s):
            A, B, Aq, Bq = hpools[li % nshape]
            n_all, X, Y = (chunk, A, B) if role == "train" else (Nq, Aq, Bq)
            return [(X[:min(Ph, n_all - r)], Y[:min(Ph, n_all - r)], r, min(Ph, n_all - r)) for r in range(0, n_all, Ph)]

        # the H2D ceiling, measured as the e2e leg copies: four copy streams at once, several GB
        copy_streams = [torch.cuda.Stream(device=dev) for _ in range(4)]
        srcs = [hpools[si][i] for si in range(nshape) for i in range(2)]
        while len(srcs) > 2 and sum(x.numel() * 2 for x in srcs) > 12e9:
            srcs = srcs[:-1]
        dsts = [torch.empty_like(x, device=dev) for x in srcs]
        nbytes = sum(x.numel() * 2 for x in srcs)
        h2d_gbs = 0.0
        for rep in range(4):  # best of four: the link's ceiling, not a slow first pass
            torch.cuda.synchronize()
            c0 = time.perf_counter()
            for i, (hs, ds) in enumerate(zip(srcs, dsts)):
                with torch.cuda.stream(copy_streams[i % 4]):
                    ds.copy_(hs, non_blocking=True)
            torch.cuda.synchronize()
            h2d_gbs = max(h2d_gbs, nbytes / (time.perf_counter() - c0) / 1e9)
        del dsts
        idx_h = torch.empty((Nq, args.topk), dtype=torch.int32).pin_memory()
        val_h = torch.empty((Nq, args.topk), dtype=torch.float32).pin_memory()

        def e2e_step():
            s = state["s"]
            advance(host_factors)
            job.join()
            r0, r1 = job.share(s, Nq)
            idx_h[r0:r1].copy_(job.idx[r0:r1], non_blocking=True)
            val_h[r0:r1].copy_(job.val[r0:r1], non_blocking=True)
            stream.synchronize()

        e2e_step()
        torch.cuda.synchronize()
        n_e2e = max(1, args.e2e_steps)
        if dist:
            dist.barrier()
        c0 = time.perf_counter()
        for _ in range(n_e2e):
            e2e_step()
        e2e_s = max_over_ranks((time.perf_counter() - c0) / n_e2e)
        tda.tda_device_status()
        h2d = (chunk * T * sum(di + do for di, do in linears) * 2
               + Nq * T * sum(di + do for di, do in linears) * 2 // C)
        e2e = {"value": world * chunk / e2e_s, "unit": "examples/s", "h2d_bytes_per_step": world * h2d,
               "d2h_bytes_per_step": (Nq // C) * args.topk * 8, "ms_per_step": e2e_s * 1e3, "steps": n_e2e,
               "host_pool_examples": Ph, "h2d_gbs_measured_4_streams": h2d_gbs,
               "h2d_gbs_achieved": h2d / e2e_s / 1e9,
               "h2d_bound_examples_per_s": chunk / (h2d / (h2d_gbs * 1e9)), "host_numa_node": numa}
        if world > 1:
            e2e["d2h_bytes_per_step"] *= world
            e2e["note"] = "per-rank H2D figures; value and bytes summed over the replicas"
        if saved_aff is not None:
            os.sched_setaffinity(0, saved_aff)

    cpu = None
    if not args.no_cpu_baseline and rank == 0:
        def factors_of(role, li, n):
            A, B, Aq, Bq = pools[li]
            X, Y = (A, B) if role == "train" else (Aq, Bq)
            return (X[:n].float().cpu().numpy().astype(np.float64), Y[:n].float().cpu().numpy().astype(np.float64))

        v, cores, sample, _ = stack_oracle_sample(spec, factors_of)
        cpu = {"value": v, "unit": "examples/s", "cores": cores, "kind": "oracle", "sample": sample}

    line = {
        "metric": METRIC, "value": value, "unit": "examples/s", "n_gpus": world, "steps": steps,
        "warmup": args.warmup, "ms_per_step": ms, "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
        "dtype": "bf16", "data": "synthetic", "config": stack_config(args, spec), "roofline": roofline,
        "phases": phases, "cpu_baseline": cpu, "e2e": e2e, "gpu_launches": launches, "clocks": ck,
        "host_enqueue_ms_per_step": host_ms,
    }
    if rank == 0:
        print(json.dumps(line), flush=True)
    if dist:
        dist.barrier()
        dist.destroy_process_group()
    return 0


def main():
    args = parse_args()
    if args.workload in STACKS:
        if args.impl == "reference":
            return stack_reference_main(args, STACKS[args.workload])
        if args.profile_project or args.profile_precond:
            return stack_profile_main(args, STACKS[args.workload])
        return stack_main(args, STACKS[args.workload])
    if args.impl == "reference":
        return reference_main(args)
    if args.route_sweep:
        return route_sweep_main(args)
    if args.token_scores or args.masks:
        return reuse_main(args)

    import numpy as np
    import torch

    import paper_2609_38767_gb300 as tda
    from paper_2609_38767_gb300 import build as tbuild
    from paper_2609_38767_gb300 import synth

    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    torch.cuda.set_device(local)
    dist = None
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
    if rank == 0:
        tbuild.build()
    if dist:
        dist.barrier()
    tda.load()
    dev = torch.device("cuda", local)
    stream = torch.cuda.current_stream()
    T, N, Nq, k = args.T, args.n_train, args.n_query, args.k
    D = k * k
    nl = len(LINEARS)
    DT = D * nl
    sb = math.sqrt(1e-3)

    # ---- device-resident synthetic factors (untimed); rank r owns train examples
    # [r*N, (r+1)*N) of the job, the queries are replicated
    from paper_2609_38767_gb300 import shard

    e0 = shard.shard_offset(rank, N)
    At, Bt, Aq, Bq = [], [], [], []
    for li, (_, di, do) in enumerate(LINEARS):
        for store, n, role in ((At, N, 0), (Aq, Nq, 1)):
            x = torch.empty(n * T * di, dtype=torch.bfloat16, device=dev)
            synth.fill_device(x, synth.SEED_A, li + (synth.QUERY_STREAM_OFFSET if role else 0), n, T, di, 1.0,
                              e0=0 if role else e0, mask_p=0.01, mask_stream=1000 if role else 0)
            store.append(x)
        for store, n, role in ((Bt, N, 0), (Bq, Nq, 1)):
            x = torch.empty(n * T * do, dtype=torch.bfloat16, device=dev)
            synth.fill_device(x, synth.SEED_B, li + (synth.QUERY_STREAM_OFFSET if role else 0), n, T, do, sb,
                              e0=0 if role else e0, mask_p=0.01, mask_stream=1000 if role else 0)
            store.append(x)
    from paper_2609_38767_gb300.block import BlockPipeline

    kfac_mode = not args.no_precondition and args.curvature != "fisher"
    pipe = BlockPipeline([(di, do) for _, di, do in LINEARS], T, k, N, Nq, topk=args.topk,
                         precondition=not args.no_precondition, lambda_rel=0.1 if kfac_mode else 1e-2, device=dev,
                         curvature=args.curvature, query_streams=args.query_streams)
    layers, Phi, Q, idx, val = pipe.layers, pipe.Phi, pipe.Q, pipe.idx, pipe.val
    select = shard.device_select(tda)
    torch.cuda.synchronize()

    ev = []  # (start, end, algorithmic bytes) per projection launch of the train set
    phase_ev = []  # (name, event) marks of the timed steps

    def attribute(project, record=False):
        marks = {}

        def mark(name):
            if record:
                e = torch.cuda.Event(enable_timing=True)
                e.record(stream)
                phase_ev.append((name, e))

        def before(li):
            if record:
                e0 = torch.cuda.Event(enable_timing=True)
                e0.record(stream)
                marks[li] = e0

        def train(li, L, route, phi, ld):
            before(li)
            project("train", li, L, route, phi, ld)

        def after(li):
            if record:
                e1 = torch.cuda.Event(enable_timing=True)
                e1.record(stream)
                L = layers[li]
                ev.append((marks[li], e1, N * (T * (L.d_in + L.d_out) * 2 + 4 * D)))

        if args.project_only:
            for li, (L, route) in enumerate(zip(layers, pipe.routes())):
                train(li, L, route, Phi[:, li * D:], DT)
                after(li)
            return
        pipe.run(train, lambda li, L, route, phi, ld: project("query", li, L, route, phi, ld), after, mark,
                 overlap_sms=args.overlap_sms, dist=dist)
        if dist:
            # the exchange step of a sharded job: the global top-k from every rank's top-k
            shard.merge_topk(idx, val, e0, args.topk, dist, world, select)

    def project_dev(role, li, L, route, phi, ld):
        if role == "train" and kfac_mode:
            pipe.project_train_kfac(li, At[li], Bt[li], phi, ld)
        elif role == "train":
            tda.tda_project(L, tda.TDA_BF16, At[li], Bt[li], N, phi, ld, route)
        else:
            tda.tda_project(L, tda.TDA_BF16, Aq[li], Bq[li], Nq, phi, ld, route)

    for _ in range(args.warmup):
        attribute(project_dev)
    tda.tda_device_status()
    if dist:
        dist.barrier()
    torch.cuda.synchronize()
    clocks = ClockSampler(local)
    clocks.start()
    time.sleep(0.3)
    launches0 = tda.tda_launch_count()
    t_start, t_end = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    t_start.record(stream)
    for _ in range(args.steps):
        attribute(project_dev, record=True)
    t_end.record(stream)
    torch.cuda.synchronize()
    launches = tda.tda_launch_count() - launches0
    ck = clocks.stop()
    tda.tda_device_status()
    ms = t_start.elapsed_time(t_end) / args.steps
    if dist:
        t = torch.tensor([ms], device=dev)
        dist.all_reduce(t, op=dist.ReduceOp.MAX)
        ms = float(t.item())
        dist.barrier()
    value = world * N / (ms * 1e-3)
    proj_ms = sum(a.elapsed_time(b) for a, b, _ in ev)
    proj_bytes = sum(x for _, _, x in ev)
    peaks = {}
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            peaks = json.load(f)
    except OSError:
        pass
    hbm = float(peaks.get("hbm_gbs", 6800.0))
    achieved = proj_bytes / (proj_ms * 1e-3) / 1e9
    engines = sorted({tda.tda_project_engine(L, tda.TDA_BF16, At[li], Bt[li]) for li, L in enumerate(layers)})
    same_kernel = projection_kernel_sha256() == TRAFFIC_KERNEL_SHA256
    per_launch = proj_bytes / max(len(ev), 1)
    roofline = {"bound": "hbm", "kernel": "factored projection (train, 7 linears)",
                "engine": "tcgen05" if engines == [1] else ("cuda-core" if engines == [0] else "mixed"), "achieved": achieved,
                "peak": hbm, "unit": "GB/s", "frac": achieved / hbm,
                "traffic": (TRAFFIC_RATIO[k] * per_launch
                            if (same_kernel and engines == [1] and not kfac_mode and k in TRAFFIC_RATIO) else None),
                "algorithmic_bytes_per_launch": per_launch,
                "peak_source": "MEASURED_PEAKS.json hbm_gbs" if peaks else "fallback 6.8 TB/s",
                "share_of_step": proj_ms / (ms * args.steps)}

    # ---- every phase of the step against its own ceiling
    alu = 152 * 128 * 2 * float(peaks.get("sm_max_mhz", 2070.0)) * 1e6 / 1e12  # fp32 FMA TFLOP/s
    # 3xTF32 on the tensor cores: the sustained bf16 peak x the nominal tf32/bf16 ratio (1/2), three
    # MMAs per fp32 product: the ceiling in useful fp32 flops of the fit and the score
    tf32x3 = float(peaks.get("bf16_tflops_sustained", 1700.0)) * 0.5 / 3.0
    ph = {}
    for (name, e0), (_, e1) in zip(phase_ev, phase_ev[1:]):
        if name is not None:
            ph[name] = ph.get(name, 0.0) + e0.elapsed_time(e1) / args.steps
    Dn = float(D)
    per_unit = {
        "project_train": ("hbm", sum(N * (T * (L.d_in + L.d_out) * 2 + 4 * D) for L in layers), hbm, "GB/s"),
        "project_query": ("hbm", sum(Nq * (T * (L.d_in + L.d_out) * 2 + 4 * D) for L in layers), hbm, "GB/s"),
        "fisher_fit": ("tensor", nl * N * Dn * (Dn + 1), tf32x3, "TFLOP/s"),
        "factor": ("latency", nl * Dn ** 3 / 3, alu, "TFLOP/s"),
        "apply": ("latency", (nl * 4 * 2 * Dn * k * Nq) if kfac_mode else (nl * 2 * 2 * Dn * Dn * Nq), alu, "TFLOP/s"),
        "factor_apply": ("latency", nl * (Dn ** 3 / 3 + 2 * Dn * Dn * Nq), alu, "TFLOP/s"),
        "kfac_eigen": ("latency", nl * 2 * 10 * 4.0 * k ** 3, alu, "TFLOP/s"),
        "ekfac_eigenvalues": ("alu", nl * N * 2 * 2 * Dn * k, alu, "TFLOP/s"),
        "score": ("tensor", 2.0 * Nq * N * DT, tf32x3, "TFLOP/s"),
        "topk": ("latency", 8.0 * Nq * N * 4, hbm, "GB/s"),
        # sharded job: the curvature sums added over the ranks (NCCL all-reduce)
        "curvature_allreduce": ("latency", (nl * D * D * 4) if not kfac_mode else (nl * 2 * k * k * 8), hbm, "GB/s"),
        # overlapped query side: what is left of it after the last train projection
        "query_side_tail": ("latency", nl * 2 * 2 * Dn * Dn * Nq / nl, alu, "TFLOP/s"),
    }
    if args.overlap_sms > 0 and "project_train" in ph:
        # the train phase also carries the query projection, fit, factorisation and preconditioning
        per_unit["project_train"] = ("hbm", per_unit["project_train"][1] + per_unit["project_query"][1], hbm, "GB/s")
    phases = {}
    for name, ms_ in ph.items():
        bound, work, peak, unit = per_unit[name]
        rate = work / (ms_ * 1e-3) / (1e9 if unit == "GB/s" else 1e12)
        phases[name] = {"ms": ms_, "bound": bound, "achieved": rate, "peak": peak, "unit": unit,
                        "frac": rate / peak}

    # ---- e2e through tda_project_host with pinned host factors
    e2e = None
    if not args.no_e2e and not args.project_only and not kfac_mode:
        # pinned pools on the host memory nearest the GPU: this thread runs on the
        # GPU's NUMA node while the pools are allocated and first touched
        saved_aff, numa = bind_to_gpu_numa(local)
        P = min(args.pool, N)
        pools = []
        for li, (_, di, do) in enumerate(LINEARS):
            a = torch.empty(P * T * di, dtype=torch.bfloat16).pin_memory()
            b = torch.empty(P * T * do, dtype=torch.bfloat16).pin_memory()
            a.copy_(At[li][: P * T * di])
            b.copy_(Bt[li][: P * T * do])
            qa = torch.empty(Nq * T * di, dtype=torch.bfloat16).pin_memory()
            qb = torch.empty(Nq * T * do, dtype=torch.bfloat16).pin_memory()
            qa.copy_(Aq[li])
            qb.copy_(Bq[li])
            pools.append((a, b, qa, qb))
        wsb = 2 * P * T * max(di + do for _, di, do in LINEARS) * 2
        ws = torch.empty(wsb, dtype=torch.uint8, device=dev)
        idx_h = torch.empty((Nq, args.topk), dtype=torch.int32).pin_memory()
        val_h = torch.empty((Nq, args.topk), dtype=torch.float32).pin_memory()

        def project_host(role, li, L, route, phi, ld):
            a, b, qa, qb = pools[li]
            if role == "train":
                for e0 in range(0, N, P):
                    n = min(P, N - e0)
                    tda.tda_project_host(L, tda.TDA_BF16, a, b, n, phi[e0:], ld, ws, wsb)
            else:
                tda.tda_project_host(L, tda.TDA_BF16, qa, qb, Nq, phi, ld, ws, wsb)

        # host-streamed projections share the staging workspace: one query stream
        pipe.query_streams = 1

        def e2e_step():
            attribute(project_host)
            idx_h.copy_(idx, non_blocking=True)
            val_h.copy_(val, non_blocking=True)
            stream.synchronize()

        e2e_step()
        # raw pinned-host -> device bandwidth on this machine, the ceiling of the e2e leg
        # (best of five copies of one pool, CUDA events on the copying stream)
        hb = pools[0][0]
        db = torch.empty(hb.shape, dtype=hb.dtype, device=dev)
        h2d_gbs = 0.0
        for _ in range(5):
            c0, c1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            c0.record(stream)
            db.copy_(hb, non_blocking=True)
            c1.record(stream)
            c1.synchronize()
            h2d_gbs = max(h2d_gbs, hb.numel() * 2 / (c0.elapsed_time(c1) * 1e-3) / 1e9)
        del db
        if dist:
            dist.barrier()
        torch.cuda.synchronize()
        t0 = time.perf_counter()
        for _ in range(args.e2e_steps):
            e2e_step()
        e2e_s = (time.perf_counter() - t0) / args.e2e_steps
        if dist:
            t = torch.tensor([e2e_s], device=dev)
            dist.all_reduce(t, op=dist.ReduceOp.MAX)
            e2e_s = float(t.item())
        h2d = N * T * sum(di + do for _, di, do in LINEARS) * 2 + Nq * T * sum(di + do for _, di, do in LINEARS) * 2
        e2e = {"value": world * N / e2e_s, "unit": "examples/s", "h2d_bytes_per_step": h2d,
               "d2h_bytes_per_step": Nq * args.topk * 8, "ms_per_step": e2e_s * 1e3,
               "host_pool_examples": P, "h2d_gbs_measured": h2d_gbs,
               "h2d_bound_examples_per_s": world * N / (h2d / (h2d_gbs * 1e9)), "host_numa_node": numa}
        if saved_aff is not None:
            os.sched_setaffinity(0, saved_aff)

    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline and not args.project_only:
        def factors_of(role, li, e0, n):
            src_a, src_b = (At, Bt) if role == "train" else (Aq, Bq)
            di, do = LINEARS[li][1], LINEARS[li][2]
            a = src_a[li][e0 * T * di:(e0 + n) * T * di].float().cpu().numpy().astype(np.float64)
            b = src_b[li][e0 * T * do:(e0 + n) * T * do].float().cpu().numpy().astype(np.float64)
            return a.reshape(n, T, di), b.reshape(n, T, do)

        threads = os.cpu_count() or 1
        v, cores, sample, _ = oracle_sample(args, max(2, threads), 2, factors_of)
        cpu = {"value": v, "unit": "examples/s", "cores": cores, "kind": "oracle", "sample": sample}

    if rank == 0:
        line = {
            "metric": METRIC, "value": value, "unit": "examples/s", "n_gpus": world, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": ms, "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
            "config": workload(args),
            "ranks": world, **({"exchange": "curvature sums all-reduced, global top-k merged by all-gather"}
                               if world > 1 else {}),
            "routes": {name: {0: "factored", 1: "materialize", 2: "gram"}[r] for (name, _, _), r
                       in zip(LINEARS, pipe.routes())},
            "roofline": roofline, "phases": phases, "cpu_baseline": cpu, "e2e": e2e, "gpu_launches": launches,
            "clocks": ck,
        }
        print(json.dumps(line), flush=True)
    if dist:
        dist.destroy_process_group()
    return 0


if __name__ == "__main__":
    sys.exit(main())
