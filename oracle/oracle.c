/*
 * oracle.c -- fp64 CPU oracle (TEST INFRASTRUCTURE; see oracle.h).
 *
 * Plain loops in double precision, one definition per routine, written from
 * the paper's equations. No blocking, no fusion, no reordering beyond what the
 * definition states. OpenMP, when compiled in, only distributes independent
 * examples (or query rows) over threads.
 */
#include "oracle.h"

#include <math.h>
#include <stdlib.h>
#include <string.h>
#ifdef _OPENMP
#include <omp.h>
#endif

/* ------------------------------------------------------------------------ */
/* Threads                                                                  */
/* ------------------------------------------------------------------------ */

static int32_t g_threads = 1;

void oracle_set_threads(int32_t n) { g_threads = n < 1 ? 1 : n; }
int32_t oracle_get_threads(void) {
#ifdef _OPENMP
    return g_threads;
#else
    return 1;
#endif
}

/* ------------------------------------------------------------------------ */
/* Counter-based hash for the Rademacher maps                               */
/* ------------------------------------------------------------------------ */

/* Golden-ratio increment of SplitMix64, floor(2^64 / phi) rounded to odd. */
#define ORACLE_GAMMA 0x9E3779B97F4A7C15ULL

/* SplitMix64 output function (Steele, Lea & Flood 2014): two xor-shift-
 * multiply rounds and a final xor-shift. A bijection on 64-bit words. */
uint64_t oracle_mix64(uint64_t z) {
    z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ULL;
    z = (z ^ (z >> 27)) * 0x94D049BB133111EBULL;
    return z ^ (z >> 31);
}

uint64_t oracle_splitmix64_next(uint64_t* state) {
    *state += ORACLE_GAMMA;
    return oracle_mix64(*state);
}

/* App. A.2: the two sides of a layer's factor projection draw from distinct
 * seeds derived from one per-layer base seed. Here the per-layer base seed is
 * the hash of (seed, layer) and each side's key is the hash of (base, side). */
static uint64_t oracle_side_key(uint64_t seed, uint32_t layer, int32_t side) {
    uint64_t base = oracle_mix64(seed + ORACLE_GAMMA * ((uint64_t)layer + 1u));
    return oracle_mix64(base + ORACLE_GAMMA * ((uint64_t)(uint32_t)side + 1u));
}

/* Entry (r, c) of a side's d x k sign matrix: bit (r mod 64) of the hash of
 * the counter (c, floor(r / 64)); a set bit means -1 (App. A.2, Rademacher). */
int32_t oracle_proj_sign(uint64_t seed, uint32_t layer, int32_t side, int64_t r, int64_t c) {
    uint64_t key = oracle_side_key(seed, layer, side);
    uint64_t ctr = ((uint64_t)c << 32) | (uint64_t)(r >> 6);
    uint64_t word = oracle_mix64(key + ORACLE_GAMMA * (ctr + 1u));
    return ((word >> (r & 63)) & 1u) ? -1 : 1;
}

void oracle_proj_entries(uint64_t seed, uint32_t layer, int32_t side, int32_t kind,
                         int64_t rows, int64_t cols, int8_t* out) {
    for (int64_t r = 0; r < rows; ++r)
        for (int64_t c = 0; c < cols; ++c)
            out[r * cols + c] = (int8_t)(kind == 1 ? (r == c ? 1 : 0)
                                                   : oracle_proj_sign(seed, layer, side, r, c));
}

/* App. A.2: a Rademacher map has entries +-1/sqrt(d_out), d_out being the
 * map's OUTPUT dimension, here the number of columns k of P (d x k). */
void oracle_proj_matrix(uint64_t seed, uint32_t layer, int32_t side, int32_t kind,
                        int64_t rows, int64_t cols, double* P) {
    double scale = 1.0 / sqrt((double)cols);
    for (int64_t r = 0; r < rows; ++r)
        for (int64_t c = 0; c < cols; ++c) {
            if (kind == 1)
                P[r * cols + c] = (r == c) ? 1.0 : 0.0;
            else
                P[r * cols + c] = scale * (double)oracle_proj_sign(seed, layer, side, r, c);
        }
}

/* ------------------------------------------------------------------------ */
/* Eq. 1 and Eq. 2                                                          */
/* ------------------------------------------------------------------------ */

/* Eq. 1: DW = g a^T, i.e. G[r][c] = sum over tokens t of g_t[r] a_t[c]. */
void oracle_materialize(int64_t T, int64_t d_in, int64_t d_out,
                        const double* A, const double* B, double* G) {
    for (int64_t r = 0; r < d_out; ++r)
        for (int64_t c = 0; c < d_in; ++c) {
            double s = 0.0;
            for (int64_t t = 0; t < T; ++t) s += B[t * d_out + r] * A[t * d_in + c];
            G[r * d_in + c] = s;
        }
}

/* Eq. 2: a~_t = P_a a_t, g~_t = P_g g_t, and sum_t a~_t (x) g~_t, held as the
 * k_out x k_in matrix sum_t g~_t a~_t^T. */
void oracle_project_with(int64_t T, int64_t d_in, int64_t d_out, int64_t k_in, int64_t k_out,
                         const double* P_in, const double* P_out,
                         const double* A, const double* B, double* phi) {
    double* At = (double*)malloc(sizeof(double) * (size_t)(T * k_in));
    double* Bt = (double*)malloc(sizeof(double) * (size_t)(T * k_out));
    for (int64_t t = 0; t < T; ++t) {
        for (int64_t j = 0; j < k_in; ++j) {
            double s = 0.0;
            for (int64_t c = 0; c < d_in; ++c) s += A[t * d_in + c] * P_in[c * k_in + j];
            At[t * k_in + j] = s;
        }
        for (int64_t i = 0; i < k_out; ++i) {
            double s = 0.0;
            for (int64_t r = 0; r < d_out; ++r) s += B[t * d_out + r] * P_out[r * k_out + i];
            Bt[t * k_out + i] = s;
        }
    }
    for (int64_t i = 0; i < k_out; ++i)
        for (int64_t j = 0; j < k_in; ++j) {
            double s = 0.0;
            for (int64_t t = 0; t < T; ++t) s += Bt[t * k_out + i] * At[t * k_in + j];
            phi[i * k_in + j] = s;
        }
    free(At);
    free(Bt);
}

void oracle_project_factored(int64_t N, int64_t T, int64_t d_in, int64_t d_out,
                             int64_t k_in, int64_t k_out, uint64_t seed, uint32_t layer,
                             int32_t kind, const double* A, const double* B, double* phi) {
    double* P_in = (double*)malloc(sizeof(double) * (size_t)(d_in * k_in));
    double* P_out = (double*)malloc(sizeof(double) * (size_t)(d_out * k_out));
    oracle_proj_matrix(seed, layer, 0, kind, d_in, k_in, P_in);
    oracle_proj_matrix(seed, layer, 1, kind, d_out, k_out, P_out);
#ifdef _OPENMP
#pragma omp parallel for schedule(dynamic, 1) num_threads(g_threads)
#endif
    for (int64_t n = 0; n < N; ++n)
        oracle_project_with(T, d_in, d_out, k_in, k_out, P_in, P_out,
                            A + n * T * d_in, B + n * T * d_out, phi + n * k_out * k_in);
    free(P_in);
    free(P_out);
}

/* Route (b): materialise DW (Eq. 1), then apply the same Kronecker map,
 * P_out^T G P_in, whose vec is (P_a (x) P_g) gamma (Eq. 2). */
void oracle_project_materialized(int64_t N, int64_t T, int64_t d_in, int64_t d_out,
                                 int64_t k_in, int64_t k_out, uint64_t seed, uint32_t layer,
                                 int32_t kind, const double* A, const double* B, double* phi) {
    double* P_in = (double*)malloc(sizeof(double) * (size_t)(d_in * k_in));
    double* P_out = (double*)malloc(sizeof(double) * (size_t)(d_out * k_out));
    oracle_proj_matrix(seed, layer, 0, kind, d_in, k_in, P_in);
    oracle_proj_matrix(seed, layer, 1, kind, d_out, k_out, P_out);
#ifdef _OPENMP
#pragma omp parallel for schedule(dynamic, 1) num_threads(g_threads)
#endif
    for (int64_t n = 0; n < N; ++n) {
        double* G = (double*)malloc(sizeof(double) * (size_t)(d_out * d_in));
        double* X = (double*)malloc(sizeof(double) * (size_t)(d_out * k_in));
        oracle_materialize(T, d_in, d_out, A + n * T * d_in, B + n * T * d_out, G);
        for (int64_t r = 0; r < d_out; ++r)
            for (int64_t j = 0; j < k_in; ++j) {
                double s = 0.0;
                for (int64_t c = 0; c < d_in; ++c) s += G[r * d_in + c] * P_in[c * k_in + j];
                X[r * k_in + j] = s;
            }
        double* out = phi + n * k_out * k_in;
        for (int64_t i = 0; i < k_out; ++i)
            for (int64_t j = 0; j < k_in; ++j) {
                double s = 0.0;
                for (int64_t r = 0; r < d_out; ++r) s += P_out[r * k_out + i] * X[r * k_in + j];
                out[i * k_in + j] = s;
            }
        free(G);
        free(X);
    }
    free(P_in);
    free(P_out);
}

/* ------------------------------------------------------------------------ */
/* Unprojected similarity                                                   */
/* ------------------------------------------------------------------------ */

/* <DW_q, DW_i>_F with both gradients materialised by Eq. 1. */
void oracle_similarity_materialized(int64_t T, int64_t d_in, int64_t d_out,
                                    int64_t n_q, const double* Aq, const double* Bq,
                                    int64_t n_t, const double* At, const double* Bt, double* S) {
    size_t gsz = (size_t)(d_out * d_in);
    double* Gq = (double*)malloc(sizeof(double) * gsz * (size_t)n_q);
    double* Gt = (double*)malloc(sizeof(double) * gsz * (size_t)n_t);
    for (int64_t q = 0; q < n_q; ++q)
        oracle_materialize(T, d_in, d_out, Aq + q * T * d_in, Bq + q * T * d_out, Gq + q * gsz);
#ifdef _OPENMP
#pragma omp parallel for schedule(dynamic, 1) num_threads(g_threads)
#endif
    for (int64_t i = 0; i < n_t; ++i)
        oracle_materialize(T, d_in, d_out, At + i * T * d_in, Bt + i * T * d_out, Gt + i * gsz);
    for (int64_t q = 0; q < n_q; ++q)
        for (int64_t i = 0; i < n_t; ++i) {
            double s = 0.0;
            for (size_t e = 0; e < gsz; ++e) s += Gq[q * gsz + e] * Gt[i * gsz + e];
            S[q * n_t + i] = s;
        }
    free(Gq);
    free(Gt);
}

/* Eq. 4: <gamma_q, gamma_i> = sum_t sum_s <a_t^q, a_s^i> <g_t^q, g_s^i>. */
void oracle_similarity_gram(int64_t T, int64_t d_in, int64_t d_out,
                            int64_t n_q, const double* Aq, const double* Bq,
                            int64_t n_t, const double* At, const double* Bt, double* S) {
#ifdef _OPENMP
#pragma omp parallel for schedule(dynamic, 1) num_threads(g_threads)
#endif
    for (int64_t i = 0; i < n_t; ++i)
        for (int64_t q = 0; q < n_q; ++q) {
            const double* aq = Aq + q * T * d_in;
            const double* bq = Bq + q * T * d_out;
            const double* ai = At + i * T * d_in;
            const double* bi = Bt + i * T * d_out;
            double s = 0.0;
            for (int64_t t = 0; t < T; ++t)
                for (int64_t u = 0; u < T; ++u) {
                    double aa = 0.0, bb = 0.0;
                    for (int64_t c = 0; c < d_in; ++c) aa += aq[t * d_in + c] * ai[u * d_in + c];
                    for (int64_t r = 0; r < d_out; ++r) bb += bq[t * d_out + r] * bi[u * d_out + r];
                    s += aa * bb;
                }
            S[q * n_t + i] = s;
        }
}

/* ------------------------------------------------------------------------ */
/* Norms and cosine                                                         */
/* ------------------------------------------------------------------------ */

void oracle_sq_norms_materialized(int64_t N, int64_t T, int64_t d_in, int64_t d_out,
                                  const double* A, const double* B, double* out) {
#ifdef _OPENMP
#pragma omp parallel for schedule(dynamic, 1) num_threads(g_threads)
#endif
    for (int64_t n = 0; n < N; ++n) {
        double* G = (double*)malloc(sizeof(double) * (size_t)(d_out * d_in));
        oracle_materialize(T, d_in, d_out, A + n * T * d_in, B + n * T * d_out, G);
        double s = 0.0;
        for (int64_t e = 0; e < d_out * d_in; ++e) s += G[e] * G[e];
        out[n] = s;
        free(G);
    }
}

void oracle_sq_norms_gram(int64_t N, int64_t T, int64_t d_in, int64_t d_out,
                          const double* A, const double* B, double* out) {
    for (int64_t n = 0; n < N; ++n)
        oracle_similarity_gram(T, d_in, d_out, 1, A + n * T * d_in, B + n * T * d_out,
                               1, A + n * T * d_in, B + n * T * d_out, out + n);
}

/* LESS-style cosine: the inner product over the product of the two norms. */
void oracle_cosine(int64_t n_q, int64_t n_t, const double* S, const double* nq,
                   const double* nt, double* C) {
    for (int64_t q = 0; q < n_q; ++q)
        for (int64_t i = 0; i < n_t; ++i)
            C[q * n_t + i] = S[q * n_t + i] / sqrt(nq[q] * nt[i]);
}

/* ------------------------------------------------------------------------ */
/* Preconditioning                                                          */
/* ------------------------------------------------------------------------ */

/* Empirical Fisher of the projected training gradients, the mean of the
 * outer products phi_i phi_i^T over the N training examples. Entry (a, b) is
 * the sum over n = 0..N-1, in that order, of phi_na phi_nb, divided by N; the
 * loop over n sits outside the loop over b only so that the rows of phi are
 * read contiguously (each entry's additions happen in the same order). */
void oracle_fisher(int64_t D, int64_t N, const double* phi, double* F) {
#ifdef _OPENMP
#pragma omp parallel for schedule(dynamic, 1) num_threads(g_threads)
#endif
    for (int64_t a = 0; a < D; ++a) {
        double* row = F + a * D;
        for (int64_t b = 0; b < D; ++b) row[b] = 0.0;
        for (int64_t n = 0; n < N; ++n) {
            const double pa = phi[n * D + a];
            for (int64_t b = 0; b < D; ++b) row[b] += pa * phi[n * D + b];
        }
        for (int64_t b = 0; b < D; ++b) row[b] = row[b] / (double)N;
    }
}

/* Damping in units of the mean eigenvalue (App. B.2); the mean eigenvalue of a
 * symmetric matrix is its trace over its order. */
double oracle_damping(int64_t D, const double* F, double lambda_abs, double lambda_rel) {
    double tr = 0.0;
    for (int64_t a = 0; a < D; ++a) tr += F[a * D + a];
    return lambda_abs + lambda_rel * tr / (double)D;
}

/* The same damping from the features themselves, without forming F: the
 * diagonal entry F_aa is (sum over n of phi_na^2) / N, summed over a in order
 * (the same additions as oracle_fisher followed by oracle_damping). */
double oracle_damping_features(int64_t D, int64_t N, const double* phi, double lambda_abs,
                               double lambda_rel) {
    double tr = 0.0;
    for (int64_t a = 0; a < D; ++a) {
        double s = 0.0;
        for (int64_t n = 0; n < N; ++n) s += phi[n * D + a] * phi[n * D + a];
        tr += s / (double)N;
    }
    return lambda_abs + lambda_rel * tr / (double)D;
}

/* Textbook Cholesky-Banachiewicz: L[j][j] = sqrt(M[j][j] - sum_k L[j][k]^2),
 * L[i][j] = (M[i][j] - sum_k L[i][k] L[j][k]) / L[j][j] for i > j. */
int32_t oracle_cholesky(int64_t D, double* M) {
    for (int64_t j = 0; j < D; ++j) {
        double s = M[j * D + j];
        for (int64_t k = 0; k < j; ++k) s -= M[j * D + k] * M[j * D + k];
        if (!(s > 0.0)) return (int32_t)(j + 1);
        double ljj = sqrt(s);
        M[j * D + j] = ljj;
        /* for a fixed column j the rows i > j are independent of each other */
#ifdef _OPENMP
#pragma omp parallel for schedule(static) num_threads(g_threads) if (D - j > 256)
#endif
        for (int64_t i = j + 1; i < D; ++i) {
            double t = M[i * D + j];
            for (int64_t k = 0; k < j; ++k) t -= M[i * D + k] * M[j * D + k];
            M[i * D + j] = t / ljj;
        }
    }
    for (int64_t i = 0; i < D; ++i)
        for (int64_t j = i + 1; j < D; ++j) M[i * D + j] = 0.0;
    return 0;
}

/* Per-layer preconditioning of the queries (App. B.3): with
 * F + lambda I = L L^T, solve L y = q by forward and L^T x = y by backward
 * substitution, so x = (F + lambda I)^{-1} q. Query rows are independent. */
int32_t oracle_precondition(int64_t D, const double* F, double lambda,
                            int64_t n_q, const double* Q, double* Qhat) {
    double* L = (double*)malloc(sizeof(double) * (size_t)(D * D));
    memcpy(L, F, sizeof(double) * (size_t)(D * D));
    for (int64_t a = 0; a < D; ++a) L[a * D + a] += lambda;
    int32_t st = oracle_cholesky(D, L);
    if (st != 0) {
        free(L);
        return st;
    }
#ifdef _OPENMP
#pragma omp parallel for schedule(dynamic, 1) num_threads(g_threads)
#endif
    for (int64_t q = 0; q < n_q; ++q) {
        double* y = (double*)malloc(sizeof(double) * (size_t)D);
        const double* b = Q + q * D;
        double* x = Qhat + q * D;
        for (int64_t i = 0; i < D; ++i) {
            double s = b[i];
            for (int64_t k = 0; k < i; ++k) s -= L[i * D + k] * y[k];
            y[i] = s / L[i * D + i];
        }
        for (int64_t i = D - 1; i >= 0; --i) {
            double s = y[i];
            for (int64_t k = i + 1; k < D; ++k) s -= L[k * D + i] * x[k];
            x[i] = s / L[i * D + i];
        }
        free(y);
    }
    free(L);
    return 0;
}

/* The same damped inverse when the Fisher has fewer examples than features
 * (N < D), without the D x D matrix. F + lambda I = lambda I + Phi^T Phi / N,
 * and the Woodbury identity gives
 *   (F + lambda I)^{-1} q = (q - Phi^T z) / lambda,
 *   (N lambda I + Phi Phi^T) z = Phi q,
 * an N x N system (Cholesky as above). Exact for any N; cheaper when N < D. */
int32_t oracle_precondition_lowrank(int64_t D, int64_t N, const double* phi, double lambda,
                                    int64_t n_q, const double* Q, double* Qhat) {
    double* K = (double*)malloc(sizeof(double) * (size_t)(N * N));
#ifdef _OPENMP
#pragma omp parallel for schedule(dynamic, 1) num_threads(g_threads)
#endif
    for (int64_t i = 0; i < N; ++i)
        for (int64_t j = 0; j < N; ++j) {
            double s = 0.0;
            for (int64_t a = 0; a < D; ++a) s += phi[i * D + a] * phi[j * D + a];
            K[i * N + j] = s;
        }
    for (int64_t i = 0; i < N; ++i) K[i * N + i] += (double)N * lambda;
    int32_t st = oracle_cholesky(N, K);
    if (st != 0) {
        free(K);
        return st;
    }
#ifdef _OPENMP
#pragma omp parallel for schedule(dynamic, 1) num_threads(g_threads)
#endif
    for (int64_t q = 0; q < n_q; ++q) {
        double* u = (double*)malloc(sizeof(double) * (size_t)N);
        double* z = (double*)malloc(sizeof(double) * (size_t)N);
        const double* b = Q + q * D;
        double* x = Qhat + q * D;
        for (int64_t i = 0; i < N; ++i) {
            double s = 0.0;
            for (int64_t a = 0; a < D; ++a) s += phi[i * D + a] * b[a];
            u[i] = s;
        }
        for (int64_t i = 0; i < N; ++i) {
            double s = u[i];
            for (int64_t k = 0; k < i; ++k) s -= K[i * N + k] * z[k];
            z[i] = s / K[i * N + i];
        }
        for (int64_t i = N - 1; i >= 0; --i) {
            double s = z[i];
            for (int64_t k = i + 1; k < N; ++k) s -= K[k * N + i] * z[k];
            z[i] = s / K[i * N + i];
        }
        for (int64_t a = 0; a < D; ++a) {
            double s = b[a];
            for (int64_t i = 0; i < N; ++i) s -= phi[i * D + a] * z[i];
            x[a] = s / lambda;
        }
        free(u);
        free(z);
    }
    free(K);
    return 0;
}

/* ------------------------------------------------------------------------ */
/* Kronecker-factored curvature on projected factors                        */
/* ------------------------------------------------------------------------ */

void oracle_kfac_covariances(int64_t N, int64_t T, int64_t d_in, int64_t d_out,
                             int64_t k_in, int64_t k_out, uint64_t seed, uint32_t layer,
                             int32_t kind, const double* A, const double* B,
                             double* Ca, double* Cg) {
    double* P_in = (double*)malloc(sizeof(double) * (size_t)(d_in * k_in));
    double* P_out = (double*)malloc(sizeof(double) * (size_t)(d_out * k_out));
    oracle_proj_matrix(seed, layer, 0, kind, d_in, k_in, P_in);
    oracle_proj_matrix(seed, layer, 1, kind, d_out, k_out, P_out);
    /* per-example sums first (examples in parallel), then their sum in example order */
    double* pa = (double*)calloc((size_t)(N > 0 ? N : 1) * (size_t)(k_in * k_in), sizeof(double));
    double* pg = (double*)calloc((size_t)(N > 0 ? N : 1) * (size_t)(k_out * k_out), sizeof(double));
#ifdef _OPENMP
#pragma omp parallel for schedule(dynamic, 1) num_threads(g_threads)
#endif
    for (int64_t n = 0; n < N; ++n) {
        const double* An = A + n * T * d_in;
        const double* Bn = B + n * T * d_out;
        double* at = (double*)malloc(sizeof(double) * (size_t)k_in);
        double* gt = (double*)malloc(sizeof(double) * (size_t)k_out);
        for (int64_t t = 0; t < T; ++t) {
            for (int64_t j = 0; j < k_in; ++j) {
                double s = 0.0;
                for (int64_t c = 0; c < d_in; ++c) s += An[t * d_in + c] * P_in[c * k_in + j];
                at[j] = s;
            }
            for (int64_t i = 0; i < k_out; ++i) {
                double s = 0.0;
                for (int64_t r = 0; r < d_out; ++r) s += Bn[t * d_out + r] * P_out[r * k_out + i];
                gt[i] = s;
            }
            for (int64_t j = 0; j < k_in; ++j)
                for (int64_t j2 = 0; j2 < k_in; ++j2) pa[n * k_in * k_in + j * k_in + j2] += at[j] * at[j2];
            for (int64_t i = 0; i < k_out; ++i)
                for (int64_t i2 = 0; i2 < k_out; ++i2) pg[n * k_out * k_out + i * k_out + i2] += gt[i] * gt[i2];
        }
        free(at);
        free(gt);
    }
    const double M = (double)N * (double)T;
    for (int64_t e = 0; e < k_in * k_in; ++e) {
        double s = 0.0;
        for (int64_t n = 0; n < N; ++n) s += pa[n * k_in * k_in + e];
        Ca[e] = M > 0 ? s / M : 0.0;
    }
    for (int64_t e = 0; e < k_out * k_out; ++e) {
        double s = 0.0;
        for (int64_t n = 0; n < N; ++n) s += pg[n * k_out * k_out + e];
        Cg[e] = M > 0 ? s / M : 0.0;
    }
    free(pa);
    free(pg);
    free(P_in);
    free(P_out);
}

/* Cyclic Jacobi: sweep the pairs (p, q), p < q, in row order; each rotation
 * J(p, q, theta) zeroes the (p, q) entry of A <- J^T A J, and V <- V J
 * accumulates the eigenvectors. Stop once the off-diagonal Frobenius norm is
 * at most 1e-15 of the matrix's. */
int32_t oracle_sym_eig(int64_t n, const double* C, double* w, double* U) {
    double* A = (double*)malloc(sizeof(double) * (size_t)(n * n > 0 ? n * n : 1));
    memcpy(A, C, sizeof(double) * (size_t)(n * n));
    for (int64_t i = 0; i < n; ++i)
        for (int64_t j = 0; j < n; ++j) U[i * n + j] = i == j ? 1.0 : 0.0;
    double fro = 0.0;
    for (int64_t e = 0; e < n * n; ++e) fro += A[e] * A[e];
    int32_t sweeps = -1;
    for (int32_t sweep = 0; sweep <= 100; ++sweep) {
        double off = 0.0;
        for (int64_t i = 0; i < n; ++i)
            for (int64_t j = 0; j < n; ++j)
                if (i != j) off += A[i * n + j] * A[i * n + j];
        if (off <= 1e-30 * fro) {
            sweeps = sweep;
            break;
        }
        if (sweep == 100) break;
        for (int64_t p = 0; p < n - 1; ++p)
            for (int64_t q = p + 1; q < n; ++q) {
                const double apq = A[p * n + q];
                if (apq == 0.0) continue;
                /* tan(theta) as the smaller root of t^2 + 2 tau t - 1 = 0 */
                const double tau = (A[q * n + q] - A[p * n + p]) / (2.0 * apq);
                const double t = (tau >= 0 ? 1.0 : -1.0) / (fabs(tau) + sqrt(1.0 + tau * tau));
                const double c = 1.0 / sqrt(1.0 + t * t), s = t * c;
                for (int64_t k = 0; k < n; ++k) { /* A <- A J (columns p, q) */
                    const double akp = A[k * n + p], akq = A[k * n + q];
                    A[k * n + p] = c * akp - s * akq;
                    A[k * n + q] = s * akp + c * akq;
                }
                for (int64_t k = 0; k < n; ++k) { /* A <- J^T A (rows p, q) */
                    const double apk = A[p * n + k], aqk = A[q * n + k];
                    A[p * n + k] = c * apk - s * aqk;
                    A[q * n + k] = s * apk + c * aqk;
                }
                for (int64_t k = 0; k < n; ++k) { /* V <- V J */
                    const double vkp = U[k * n + p], vkq = U[k * n + q];
                    U[k * n + p] = c * vkp - s * vkq;
                    U[k * n + q] = s * vkp + c * vkq;
                }
            }
    }
    /* sort ascending (selection sort), permuting eigenvector columns along */
    for (int64_t i = 0; i < n; ++i) w[i] = A[i * n + i];
    for (int64_t i = 0; i < n; ++i) {
        int64_t m = i;
        for (int64_t j = i + 1; j < n; ++j)
            if (w[j] < w[m]) m = j;
        if (m != i) {
            const double tw = w[i];
            w[i] = w[m];
            w[m] = tw;
            for (int64_t k = 0; k < n; ++k) {
                const double tu = U[k * n + i];
                U[k * n + i] = U[k * n + m];
                U[k * n + m] = tu;
            }
        }
    }
    free(A);
    return sweeps;
}

void oracle_kfac_eigenvalues(int64_t k_in, int64_t k_out, const double* wa, const double* wg,
                             double* Lam) {
    for (int64_t r = 0; r < k_out; ++r)
        for (int64_t c = 0; c < k_in; ++c) Lam[r * k_in + c] = wg[r] * wa[c];
}

/* X = Ug^T V Ua for one k_out x k_in matrix V */
static void to_eigenbasis(int64_t k_in, int64_t k_out, const double* Ua, const double* Ug,
                          const double* V, double* X) {
    double* Y = (double*)malloc(sizeof(double) * (size_t)(k_out * k_in));
    for (int64_t r = 0; r < k_out; ++r) /* Y = V Ua */
        for (int64_t c = 0; c < k_in; ++c) {
            double s = 0.0;
            for (int64_t j = 0; j < k_in; ++j) s += V[r * k_in + j] * Ua[j * k_in + c];
            Y[r * k_in + c] = s;
        }
    for (int64_t r = 0; r < k_out; ++r) /* X = Ug^T Y */
        for (int64_t c = 0; c < k_in; ++c) {
            double s = 0.0;
            for (int64_t i = 0; i < k_out; ++i) s += Ug[i * k_out + r] * Y[i * k_in + c];
            X[r * k_in + c] = s;
        }
    free(Y);
}

void oracle_ekfac_eigenvalues(int64_t N, int64_t k_in, int64_t k_out, const double* phi,
                              const double* Ua, const double* Ug, double* Lam) {
    const int64_t D = k_in * k_out;
    double* X = (double*)malloc(sizeof(double) * (size_t)((N > 0 ? N : 1) * D));
#ifdef _OPENMP
#pragma omp parallel for schedule(dynamic, 1) num_threads(g_threads)
#endif
    for (int64_t n = 0; n < N; ++n) to_eigenbasis(k_in, k_out, Ua, Ug, phi + n * D, X + n * D);
    for (int64_t e = 0; e < D; ++e) {
        double s = 0.0;
        for (int64_t n = 0; n < N; ++n) s += X[n * D + e] * X[n * D + e];
        Lam[e] = N > 0 ? s / (double)N : 0.0;
    }
    free(X);
}

double oracle_kfac_damping(int64_t k_in, int64_t k_out, const double* Lam, double lambda_abs,
                           double lambda_rel) {
    double s = 0.0;
    for (int64_t e = 0; e < k_in * k_out; ++e) s += Lam[e];
    return lambda_abs + lambda_rel * s / (double)(k_in * k_out);
}

void oracle_kfac_precondition(int64_t k_in, int64_t k_out, const double* Ua, const double* Ug,
                              const double* Lam, double lambda, int64_t n_q, const double* Q,
                              double* Qhat) {
    const int64_t D = k_in * k_out;
#ifdef _OPENMP
#pragma omp parallel for schedule(dynamic, 1) num_threads(g_threads)
#endif
    for (int64_t q = 0; q < n_q; ++q) {
        double* X = (double*)malloc(sizeof(double) * (size_t)D);
        double* Y = (double*)malloc(sizeof(double) * (size_t)D);
        to_eigenbasis(k_in, k_out, Ua, Ug, Q + q * D, X);
        for (int64_t e = 0; e < D; ++e) X[e] /= Lam[e] + lambda;
        for (int64_t r = 0; r < k_out; ++r) /* Y = X Ua^T */
            for (int64_t c = 0; c < k_in; ++c) {
                double s = 0.0;
                for (int64_t j = 0; j < k_in; ++j) s += X[r * k_in + j] * Ua[c * k_in + j];
                Y[r * k_in + c] = s;
            }
        for (int64_t r = 0; r < k_out; ++r) /* Qhat = Ug Y */
            for (int64_t c = 0; c < k_in; ++c) {
                double s = 0.0;
                for (int64_t i = 0; i < k_out; ++i) s += Ug[r * k_out + i] * Y[i * k_in + c];
                Qhat[q * D + r * k_in + c] = s;
            }
        free(X);
        free(Y);
    }
}

/* ------------------------------------------------------------------------ */
/* Token-level scores and random-mask reduction                             */
/* ------------------------------------------------------------------------ */

void oracle_token_scores(int64_t N, int64_t T, int64_t d_in, int64_t d_out, int64_t k_in,
                         int64_t k_out, uint64_t seed, uint32_t layer, int32_t kind,
                         const double* A, const double* B, int64_t n_q, const double* R,
                         double* out) {
    double* P_in = (double*)malloc(sizeof(double) * (size_t)(d_in * k_in));
    double* P_out = (double*)malloc(sizeof(double) * (size_t)(d_out * k_out));
    oracle_proj_matrix(seed, layer, 0, kind, d_in, k_in, P_in);
    oracle_proj_matrix(seed, layer, 1, kind, d_out, k_out, P_out);
#ifdef _OPENMP
#pragma omp parallel for schedule(dynamic, 1) num_threads(g_threads)
#endif
    for (int64_t n = 0; n < N; ++n) {
        double* at = (double*)malloc(sizeof(double) * (size_t)k_in);
        double* gt = (double*)malloc(sizeof(double) * (size_t)k_out);
        for (int64_t t = 0; t < T; ++t) {
            const double* a = A + (n * T + t) * d_in;
            const double* g = B + (n * T + t) * d_out;
            for (int64_t c = 0; c < k_in; ++c) { /* a~_t = P_a a_t */
                double s = 0.0;
                for (int64_t x = 0; x < d_in; ++x) s += a[x] * P_in[x * k_in + c];
                at[c] = s;
            }
            for (int64_t r = 0; r < k_out; ++r) { /* g~_t = P_g g_t */
                double s = 0.0;
                for (int64_t x = 0; x < d_out; ++x) s += g[x] * P_out[x * k_out + r];
                gt[r] = s;
            }
            for (int64_t j = 0; j < n_q; ++j) { /* g~_t^T R_j a~_t */
                const double* Rj = R + j * k_out * k_in;
                double s = 0.0;
                for (int64_t r = 0; r < k_out; ++r) {
                    double u = 0.0;
                    for (int64_t c = 0; c < k_in; ++c) u += Rj[r * k_in + c] * at[c];
                    s += gt[r] * u;
                }
                out[(j * N + n) * T + t] = s;
            }
        }
        free(at);
        free(gt);
    }
    free(P_in);
    free(P_out);
}

void oracle_mask_gather(int64_t N, int64_t T, int64_t d_in, int64_t d_out, const double* A,
                        const double* B, int64_t n_coords, const int32_t* rows,
                        const int32_t* cols, double* out) {
#ifdef _OPENMP
#pragma omp parallel for schedule(dynamic, 1) num_threads(g_threads)
#endif
    for (int64_t n = 0; n < N; ++n)
        for (int64_t m = 0; m < n_coords; ++m) {
            double s = 0.0;
            for (int64_t t = 0; t < T; ++t)
                s += B[(n * T + t) * d_out + rows[m]] * A[(n * T + t) * d_in + cols[m]];
            out[n * n_coords + m] = s;
        }
}

/* ------------------------------------------------------------------------ */
/* Scores and top-k                                                         */
/* ------------------------------------------------------------------------ */

/* Gradient inner products between (preconditioned) queries and training
 * features, the GradDot score when Qhat = Q (Sec. 3.2, Eq. 4's left side). */
void oracle_score(int64_t n_q, int64_t n_t, int64_t D,
                  const double* Qhat, const double* phi, double* S) {
#ifdef _OPENMP
#pragma omp parallel for schedule(dynamic, 1) num_threads(g_threads)
#endif
    for (int64_t q = 0; q < n_q; ++q)
        for (int64_t i = 0; i < n_t; ++i) {
            double s = 0.0;
            for (int64_t f = 0; f < D; ++f) s += Qhat[q * D + f] * phi[i * D + f];
            S[q * n_t + i] = s;
        }
}

typedef struct {
    double v;
    int32_t i;
} oracle_pair;

/* Descending value, then ascending index, with NaN above every number (NaNs
 * ordered by index among themselves) and -0 equal to +0 (IEEE comparison):
 * a total order, so qsort's result is the unique sorted sequence. */
static int oracle_pair_cmp(const void* x, const void* y) {
    const oracle_pair* a = (const oracle_pair*)x;
    const oracle_pair* b = (const oracle_pair*)y;
    const int na = a->v != a->v, nb = b->v != b->v;
    if (na != nb) return na ? -1 : 1;
    if (!na) {
        if (a->v > b->v) return -1;
        if (a->v < b->v) return 1;
    }
    return (a->i > b->i) - (a->i < b->i);
}

void oracle_topk(int64_t n_q, int64_t n_t, const double* S, int32_t k,
                 int32_t* idx, double* val) {
    oracle_pair* row = (oracle_pair*)malloc(sizeof(oracle_pair) * (size_t)n_t);
    for (int64_t q = 0; q < n_q; ++q) {
        for (int64_t i = 0; i < n_t; ++i) {
            row[i].v = S[q * n_t + i];
            row[i].i = (int32_t)i;
        }
        qsort(row, (size_t)n_t, sizeof(oracle_pair), oracle_pair_cmp);
        for (int32_t j = 0; j < k; ++j) {
            idx[q * k + j] = row[j].i;
            val[q * k + j] = row[j].v;
        }
    }
    free(row);
}

/* ------------------------------------------------------------------------ */
/* Route costs (App. A.4, Table 2), 2 flops per multiply-add                */
/* ------------------------------------------------------------------------ */

int32_t oracle_route_costs(int32_t op, int64_t n1, int64_t n2, int64_t T,
                           int64_t d_in, int64_t d_out, int64_t k_in, int64_t k_out,
                           double cost[3]) {
    double B1 = (double)n1, B2 = (double)n2, t = (double)T;
    double Ni = (double)d_in, No = (double)d_out, ka = (double)k_in, kg = (double)k_out;
    /* projecting one example's factors: a~ = P_a a (T x k_in), g~ = P_g g */
    double proj_factors = 2.0 * t * (Ni * ka + No * kg);
    /* contracting the projected factors over tokens into k_out x k_in */
    double contract = 2.0 * t * ka * kg;
    /* materialising DW (Eq. 1) and applying both maps to it */
    double build = 2.0 * t * Ni * No;
    double project_dense = 2.0 * No * Ni * ka + 2.0 * No * ka * kg;
    if (op == 0) {
        cost[0] = B1 * (proj_factors + contract);
        cost[1] = B1 * (build + project_dense);
        cost[2] = -1.0;
    } else if (op == 1) {
        /* Table 2 with N_i, N_o replaced by k_a, k_g, plus the shared cost of
         * projecting every example's factors. */
        cost[0] = (B1 + B2) * (proj_factors + contract) + B1 * B2 * 2.0 * ka * kg;
        cost[1] = (B1 + B2) * (build + project_dense) + B1 * B2 * 2.0 * ka * kg;
        cost[2] = (B1 + B2) * proj_factors + B1 * B2 * 2.0 * t * t * (ka + kg);
    } else if (op == 2) {
        /* Table 2 as printed: materialised vs factorised cross-Gram */
        cost[0] = -1.0;
        cost[1] = (B1 + B2) * build + B1 * B2 * 2.0 * Ni * No;
        cost[2] = B1 * B2 * 2.0 * t * t * (Ni + No);
    } else if (op == 3) {
        /* norms of projected gradients: Table 2 with B1 = B2 = 1 per example */
        cost[0] = B1 * (proj_factors + contract + 2.0 * ka * kg);
        cost[1] = B1 * (build + project_dense + 2.0 * ka * kg);
        cost[2] = B1 * (proj_factors + 2.0 * t * t * (ka + kg));
    } else {
        /* norms of unprojected gradients */
        cost[0] = -1.0;
        cost[1] = B1 * (build + 2.0 * Ni * No);
        cost[2] = B1 * 2.0 * t * t * (Ni + No);
    }
    /* cheapest valid route; ties prefer the factorised (Gram) route, then the
     * factored projection, then materialisation */
    static const int32_t pref[3] = {2, 0, 1};
    int32_t best = -1;
    for (int32_t p = 0; p < 3; ++p) {
        int32_t r = pref[p];
        if (cost[r] < 0.0) continue;
        if (best < 0 || cost[r] < cost[best]) best = r;
    }
    return best;
}
