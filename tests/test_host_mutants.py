"""The host-logic tests catch plausible mistakes in the host pipelines.

Each case plants one mistake in a copy of paper_2609_38767_gb300/stream.py
(StackJob) or block.py (BlockPipeline) -- a buffer of the wrong job, a share
boundary, a dropped accumulation, a wrong column offset or example count -- and
runs that module's CPU test (tests/test_stream_schedule_cpu.py or
tests/test_block_pipeline_cpu.py, the library calls replaced by the recording
fake) against the copy in a fresh process. The test must fail for every
mistake and pass on the unmodified copies. Mistakes live only in temporary
copies.
"""
import concurrent.futures
import os
import subprocess
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
TESTS = {"stream": "tests/test_stream_schedule_cpu.py", "block": "tests/test_block_pipeline_cpu.py"}

# (module, what the mistake is, text, the mistaken text, occurrences replaced)
MUTANTS = [
    ("stream", "query side on the other job's buffers", "        b = j % 2\n", "        b = (j + 1) % 2\n", 1),
    ("stream", "overlapping shares", "return total * s // self.C, total * (s + 1) // self.C",
     "return total * s // self.C, (total * (s + 1) + 1) // self.C", 1),
    ("stream", "top-k of the previous job instead of the one before",
     "self.topk_part(j - 2, s, mark)", "self.topk_part(j - 1, s, mark)", 2),
    ("stream", "every share overwrites the score matrix", "0.0 if l0 == 0 else 1.0", "0.0", 1),
    ("stream", "Fisher fitted over one chunk", "n=self.N, ld_phi=DT)", "n=self.chunk, ld_phi=DT)", 1),
    ("stream", "every chunk into the first rows", "Phi = self.Phi[j % 2][s * self.chunk:(s + 1) * self.chunk]",
     "Phi = self.Phi[j % 2][0:self.chunk]", 1),
    ("stream", "query features at the share's first column",
     'factors("query", li, j, s), self.Q[:, li * D:]', 'factors("query", li, j, s), self.Q[:, l0 * D:]', 1),
    ("stream", "Fisher normalised by the chunk", "st, n_total=self.N,", "st, n_total=self.chunk,", 1),
    ("stream", "score over the first linears' features", "self.Phi[b][:, l0 * D:], self.N, DT,",
     "self.Phi[b], self.N, DT,", 1),
    ("stream", "top-k rows of every share into the first rows", "self.idx[r0:], self.val[r0:]",
     "self.idx, self.val", 1),
    ("block", "score of the unpreconditioned queries", "self._score(target, mark)", "self._score(self.Q, mark)", 1),
    ("block", "train features with the leading dimension of one linear",
     "project_train(li, L, routes[li], self.Phi[:, li * D:], DT)",
     "project_train(li, L, routes[li], self.Phi[:, li * D:], D)", 2),
    ("block", "score over the first linear only", "self.Phi, self.N, DT, DT, self.S", "self.Phi, self.N, DT, D, self.S", 1),
    ("block", "absolute and relative damping swapped", "lambda_abs=self.lambda_abs, lambda_rel_mean_eig=self.lambda_rel",
     "lambda_abs=self.lambda_rel, lambda_rel_mean_eig=self.lambda_abs", 2),
    ("block", "every query projection into the first linear's columns",
     "project_query(li, L, routes[li], self.Q[:, li * D:], DT)", "project_query(li, L, routes[li], self.Q, DT)", 3),
    ("block", "Fisher fitted over half the examples", "phi=self.Phi, n=self.N, ld_phi=DT",
     "phi=self.Phi, n=self.N // 2, ld_phi=DT", 1),
]


def _run(d, module, text):
    d.mkdir()
    src = d / f"{module}.py"
    src.write_text(text)
    env = dict(os.environ, **{f"TDA_{module.upper()}_SOURCE": str(src)})
    return subprocess.run([sys.executable, "-m", "pytest", "-x", "-q", "-p", "no:cacheprovider", TESTS[module]],
                          cwd=ROOT, env=env, capture_output=True, text=True, timeout=300)


def _source(module):
    return open(os.path.join(ROOT, "paper_2609_38767_gb300", f"{module}.py")).read()


@pytest.fixture(scope="module")
def runs(tmp_path_factory):
    """Every copy's test run, several at once (each a short pytest process)."""
    import oracle
    from paper_2609_38767_gb300 import build as tbuild

    tbuild.build()  # once here, so that the concurrent runs find the libraries up to date
    oracle.build()
    jobs = {("unmodified", m): (m, _source(m)) for m in TESTS}
    for module, what, old, new, count in MUTANTS:
        src = _source(module)
        assert src.count(old) == count, f"mutation site count changed: {old}"
        jobs[(what, module)] = (module, src.replace(old, new))
    base = tmp_path_factory.mktemp("host_copies")
    with concurrent.futures.ThreadPoolExecutor(max_workers=max(1, min(8, os.cpu_count() or 1))) as ex:
        futs = {k: ex.submit(_run, base / f"copy{i}", m, t) for i, (k, (m, t)) in enumerate(jobs.items())}
        return {k: f.result() for k, f in futs.items()}


@pytest.mark.parametrize("module", sorted(TESTS))
def test_unmodified_copy_passes(runs, module):
    r = runs[("unmodified", module)]
    assert r.returncode == 0, r.stdout[-2000:] + r.stderr[-2000:]


@pytest.mark.parametrize("module,what", [m[:2] for m in MUTANTS], ids=[f"{m[0]}: {m[1]}" for m in MUTANTS])
def test_planted_mistake_fails_the_host_test(runs, module, what):
    r = runs[(what, module)]
    assert r.returncode == 1 and " failed" in r.stdout, (what, r.returncode, r.stdout[-2000:], r.stderr[-2000:])
