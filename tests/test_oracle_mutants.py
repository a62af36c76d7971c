"""The oracle's pins catch plausible mistakes in the oracle.

Each case below plants one mistake -- a dropped term, a wrong sign, index or
normalisation, a transposed operand -- in a copy of oracle/oracle.c, compiles
the copy, and runs the oracle's pin tests (tests/test_oracle_*.py: brute force,
closed forms, identities, published vectors) against it in a fresh process.
At least one pin must fail for every mistake; the unmodified copy must pass
them all. The mistakes are planted only in temporary copies, on the CPU.
"""
import concurrent.futures
import os
import shutil
import subprocess
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
ORACLE_C = os.path.join(ROOT, "oracle", "oracle.c")
PINS = ["tests/test_oracle_gradients.py", "tests/test_oracle_hash.py", "tests/test_oracle_kfac.py",
        "tests/test_oracle_precond_score.py", "tests/test_oracle_route.py", "tests/test_oracle_tokens_masks.py"]

# (what the mistake is, text in oracle.c, the mistaken text)
MUTANTS = [
    ("hash: a SplitMix64 multiplier off by one",
     "0xBF58476D1CE4E5B9ULL", "0xBF58476D1CE4E5B8ULL"),
    ("projection scale 1/sqrt(d) instead of 1/sqrt(k)",
     "double scale = 1.0 / sqrt((double)cols);", "double scale = 1.0 / sqrt((double)rows);"),
    ("Eq. 1: tokens of the two factors misaligned",
     "for (int64_t t = 0; t < T; ++t) s += B[t * d_out + r] * A[t * d_in + c];",
     "for (int64_t t = 0; t < T; ++t) s += B[t * d_out + r] * A[(T - 1 - t) * d_in + c];"),
    ("Eq. 2: feature matrix stored transposed",
     "phi[i * k_in + j] = s;", "phi[j * k_out + i] = s;"),
    ("Eq. 2: first token dropped from the contraction",
     "for (int64_t t = 0; t < T; ++t) s += Bt[t * k_out + i] * At[t * k_in + j];",
     "for (int64_t t = 1; t < T; ++t) s += Bt[t * k_out + i] * At[t * k_in + j];"),
    ("route (b): wrong column of P_in",
     "for (int64_t c = 0; c < d_in; ++c) s += G[r * d_in + c] * P_in[c * k_in + j];",
     "for (int64_t c = 0; c < d_in; ++c) s += G[r * d_in + c] * P_in[c * k_in + (k_in - 1 - j)];"),
    ("Eq. 4: only token pairs with u >= t",
     "for (int64_t u = 0; u < T; ++u) {", "for (int64_t u = t; u < T; ++u) {"),
    ("materialised similarity: last entry of DW dropped",
     "for (size_t e = 0; e < gsz; ++e) s += Gq[q * gsz + e] * Gt[i * gsz + e];",
     "for (size_t e = 0; e + 1 < gsz; ++e) s += Gq[q * gsz + e] * Gt[i * gsz + e];"),
    ("Fisher normalised by N - 1",
     "for (int64_t b = 0; b < D; ++b) row[b] = row[b] / (double)N;",
     "for (int64_t b = 0; b < D; ++b) row[b] = row[b] / (double)(N - 1);"),
    ("damping: sum of squared diagonal entries instead of the trace",
     "for (int64_t a = 0; a < D; ++a) tr += F[a * D + a];",
     "for (int64_t a = 0; a < D; ++a) tr += F[a * D + a] * F[a * D + a];"),
    ("damping from features: diagonal not divided by N",
     "tr += s / (double)N;", "tr += s;"),
    ("Cholesky: off-diagonal update with the wrong sign",
     "for (int64_t k = 0; k < j; ++k) t -= M[i * D + k] * M[j * D + k];",
     "for (int64_t k = 0; k < j; ++k) t += M[i * D + k] * M[j * D + k];"),
    ("Cholesky: last term of the diagonal sum dropped",
     "for (int64_t k = 0; k < j; ++k) s -= M[j * D + k] * M[j * D + k];",
     "for (int64_t k = 0; k + 1 < j; ++k) s -= M[j * D + k] * M[j * D + k];"),
    ("back substitution with L instead of L^T",
     "for (int64_t k = i + 1; k < D; ++k) s -= L[k * D + i] * x[k];",
     "for (int64_t k = i + 1; k < D; ++k) s -= L[i * D + k] * x[k];"),
    ("Woodbury: N lambda I written as lambda I",
     "K[i * N + i] += (double)N * lambda;", "K[i * N + i] += lambda;"),
    ("Woodbury: correction added instead of subtracted",
     "for (int64_t i = 0; i < N; ++i) s -= phi[i * D + a] * z[i];",
     "for (int64_t i = 0; i < N; ++i) s += phi[i * D + a] * z[i];"),
    ("K-FAC covariances averaged per example instead of per token",
     "const double M = (double)N * (double)T;", "const double M = (double)N;"),
    ("Jacobi rotation with the wrong sign",
     "A[k * n + p] = c * akp - s * akq;", "A[k * n + p] = c * akp + s * akq;"),
    ("EK-FAC eigenvalues: coordinates not squared",
     "for (int64_t n = 0; n < N; ++n) s += X[n * D + e] * X[n * D + e];",
     "for (int64_t n = 0; n < N; ++n) s += X[n * D + e];"),
    ("K-FAC preconditioner without the damping",
     "for (int64_t e = 0; e < D; ++e) X[e] /= Lam[e] + lambda;",
     "for (int64_t e = 0; e < D; ++e) X[e] /= Lam[e];"),
    ("eigenbasis change with U_g instead of U_g^T",
     "for (int64_t i = 0; i < k_out; ++i) s += Ug[i * k_out + r] * Y[i * k_in + c];",
     "for (int64_t i = 0; i < k_out; ++i) s += Ug[r * k_out + i] * Y[i * k_in + c];"),
    ("token scores stored example-major",
     "out[(j * N + n) * T + t] = s;", "out[(n * n_q + j) * T + t] = s;"),
    ("mask gather: tokens of the two factors misaligned",
     "s += B[(n * T + t) * d_out + rows[m]] * A[(n * T + t) * d_in + cols[m]];",
     "s += B[(n * T + t) * d_out + rows[m]] * A[(n * T + (T - 1 - t)) * d_in + cols[m]];"),
    ("cosine without the square root",
     "C[q * n_t + i] = S[q * n_t + i] / sqrt(nq[q] * nt[i]);",
     "C[q * n_t + i] = S[q * n_t + i] / (nq[q] * nt[i]);"),
    ("score: first feature dropped",
     "for (int64_t f = 0; f < D; ++f) s += Qhat[q * D + f] * phi[i * D + f];",
     "for (int64_t f = 1; f < D; ++f) s += Qhat[q * D + f] * phi[i * D + f];"),
    ("top-k: ties to the higher index",
     "return (a->i > b->i) - (a->i < b->i);", "return (a->i < b->i) - (a->i > b->i);"),
    ("top-k: NaN ranked below every number",
     "if (na != nb) return na ? -1 : 1;", "if (na != nb) return na ? 1 : -1;"),
    ("route costs: the B1 B2 2 k_a k_g term of projected similarity dropped",
     "cost[0] = (B1 + B2) * (proj_factors + contract) + B1 * B2 * 2.0 * ka * kg;",
     "cost[0] = (B1 + B2) * (proj_factors + contract);"),
    ("route costs: exact Gram route with T instead of T^2",
     "cost[2] = B1 * B2 * 2.0 * t * t * (Ni + No);", "cost[2] = B1 * B2 * 2.0 * t * (Ni + No);"),
    ("route costs: norms without the sum of squares",
     "cost[0] = B1 * (proj_factors + contract + 2.0 * ka * kg);", "cost[0] = B1 * (proj_factors + contract);"),
    ("damped inverse: lambda left off the diagonal",
     "for (int64_t a = 0; a < D; ++a) L[a * D + a] += lambda;", "for (int64_t a = 0; a < D; ++a) L[a * D + a] += 0.0;"),
    ("forward substitution without the division by the pivot",
     "y[i] = s / L[i * D + i];", "y[i] = s;"),
    ("Woodbury: final division by lambda dropped",
     "x[a] = s / lambda;", "x[a] = s;"),
    ("K-FAC eigenvalues: sum instead of product of the factors' eigenvalues",
     "Lam[r * k_in + c] = wg[r] * wa[c];", "Lam[r * k_in + c] = wg[r] + wa[c];"),
    ("EK-FAC eigenvalues: sum over the examples instead of the mean",
     "Lam[e] = N > 0 ? s / (double)N : 0.0;", "Lam[e] = N > 0 ? s : 0.0;"),
    ("K-FAC damping: mean over k_in entries instead of k_in k_out",
     "return lambda_abs + lambda_rel * s / (double)(k_in * k_out);", "return lambda_abs + lambda_rel * s / (double)k_in;"),
    ("Jacobi: eigenpairs sorted descending",
     "if (w[j] < w[m]) m = j;", "if (w[j] > w[m]) m = j;"),
    ("top-k: ascending scores",
     "if (a->v > b->v) return -1;", "if (a->v < b->v) return -1;"),
    ("route costs: projection without the token contraction",
     "cost[0] = B1 * (proj_factors + contract);", "cost[0] = B1 * proj_factors;"),
    ("route costs: exact norms by the Gram route with T instead of T^2",
     "cost[2] = B1 * 2.0 * t * t * (Ni + No);", "cost[2] = B1 * 2.0 * t * (Ni + No);"),
    ("route choice: ties prefer the factored projection over the Gram route",
     "static const int32_t pref[3] = {2, 0, 1};", "static const int32_t pref[3] = {0, 2, 1};"),
]


def _run_pins(d, source_text):
    d.mkdir()
    (d / "oracle.c").write_text(source_text)
    shutil.copy(os.path.join(ROOT, "oracle", "oracle.h"), d / "oracle.h")
    env = dict(os.environ, TDA_ORACLE_SOURCE=str(d / "oracle.c"), OMP_NUM_THREADS="2")
    return subprocess.run([sys.executable, "-m", "pytest", "-x", "-q", "-p", "no:cacheprovider", *PINS],
                          cwd=ROOT, env=env, capture_output=True, text=True, timeout=300)


@pytest.fixture(scope="module")
def runs(tmp_path_factory):
    """Every copy's pin run, several at once (each is a compile and a short pytest process)."""
    src = open(ORACLE_C).read()
    texts = {"unmodified": src}
    for what, old, new in MUTANTS:
        assert src.count(old) == 1, f"mutation site not unique or missing: {old}"
        texts[what] = src.replace(old, new)
    base = tmp_path_factory.mktemp("oracle_copies")
    with concurrent.futures.ThreadPoolExecutor(max_workers=max(1, min(8, os.cpu_count() or 1))) as ex:
        futs = {k: ex.submit(_run_pins, base / f"copy{i}", t) for i, (k, t) in enumerate(texts.items())}
        return {k: f.result() for k, f in futs.items()}


def test_unmodified_copy_passes_every_pin(runs):
    r = runs["unmodified"]
    assert r.returncode == 0, r.stdout[-2000:] + r.stderr[-2000:]


@pytest.mark.parametrize("what", [m[0] for m in MUTANTS])
def test_planted_mistake_fails_a_pin(runs, what):
    r = runs[what]
    # exit code 1: the pins ran and at least one failed (not a build or collection error)
    assert r.returncode == 1 and " failed" in r.stdout, (what, r.returncode, r.stdout[-2000:], r.stderr[-2000:])
