/*
 * oracle.h -- fp64 CPU oracle for the per-layer gradient projection, routing,
 * preconditioning and scoring path of the dattri-LLM paper.
 *
 * This is TEST INFRASTRUCTURE. Only the test suite, the smoke entry point and
 * the CPU-baseline leg of the benchmark may load or call it. It shares no code,
 * header, table or constant generator with the CUDA library; the two are
 * compared only through their outputs.
 *
 * Every routine is a plain, slow, literal transcription of a definition in the
 * paper, computed in double precision with explicit loops. Multi-example
 * routines parallelise over examples with OpenMP when it is available; each
 * example's arithmetic is sequential and in a fixed order.
 *
 * Notation (paper Sec. 3.2): a linear layer z = W a with W in R^{N_o x N_i};
 * per example the input factor a in R^{N_i x T} and output-gradient factor
 * g = Dz in R^{N_o x T}. Here an example's factors are stored token-major:
 *   A[t][c] = a_t[c]   (T x d_in,  d_in  = N_i)
 *   B[t][r] = g_t[r]   (T x d_out, d_out = N_o)
 * so that DW = g a^T has entries G[r][c] = sum_t B[t][r] A[t][c] (Eq. 1).
 * Projection maps P_a in R^{k_a x N_i}, P_g in R^{k_g x N_o} (Eq. 2) are held
 * transposed: P_in[c][j] = (P_a)[j][c] (d_in x k_in), P_out[r][i] =
 * (P_g)[i][r] (d_out x k_out). A projected feature is the k_out x k_in matrix
 * Phi = P_out^T G P_in, stored row-major (index i*k_in + j).
 *
 * Parity status: every function here is pinned by the CPU test suite (brute
 * force, closed forms, identities, published hash vectors), except where a
 * function's comment says "parity unpinned".
 */
#ifndef TDA_ORACLE_H
#define TDA_ORACLE_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* ---- counter-based hash (reading of App. A.2: per-layer, per-side seeds) ---- */

/* SplitMix64 output function (Steele, Lea & Flood, OOPSLA 2014). */
uint64_t oracle_mix64(uint64_t z);
/* One step of the SplitMix64 generator: advances *state by the golden gamma
 * and returns the mixed output. Used only to pin oracle_mix64 against the
 * generator's published reference outputs. */
uint64_t oracle_splitmix64_next(uint64_t* state);
/* Rademacher sign s in {+1,-1} of entry (r, c) of the d x k sign matrix of one
 * projection side (side 0 = input factor a, side 1 = output gradient g). */
int32_t oracle_proj_sign(uint64_t seed, uint32_t layer, int32_t side, int64_t r, int64_t c);
/* rows x cols sign matrix as int8 (kind 0 = Rademacher, 1 = identity). */
void oracle_proj_entries(uint64_t seed, uint32_t layer, int32_t side, int32_t kind,
                         int64_t rows, int64_t cols, int8_t* out);
/* rows x cols projection matrix P (App. A.2): Rademacher entries s/sqrt(cols),
 * cols = the map's output dimension; identity kind gives P = I (rows == cols). */
void oracle_proj_matrix(uint64_t seed, uint32_t layer, int32_t side, int32_t kind,
                        int64_t rows, int64_t cols, double* P);

/* ---- per-example gradients and their projections ---- */

/* Eq. 1: G[r][c] = sum_t B[t][r] A[t][c] for one example (d_out x d_in). */
void oracle_materialize(int64_t T, int64_t d_in, int64_t d_out,
                        const double* A, const double* B, double* G);

/* Eq. 2 with explicit maps, one example: At = A P_in (T x k_in),
 * Bt = B P_out (T x k_out), Phi[i][j] = sum_t Bt[t][i] At[t][j]. */
void oracle_project_with(int64_t T, int64_t d_in, int64_t d_out, int64_t k_in, int64_t k_out,
                         const double* P_in, const double* P_out,
                         const double* A, const double* B, double* phi);

/* Route (a), factored projection of N examples with the seeded maps. */
void oracle_project_factored(int64_t N, int64_t T, int64_t d_in, int64_t d_out,
                             int64_t k_in, int64_t k_out, uint64_t seed, uint32_t layer,
                             int32_t kind, const double* A, const double* B, double* phi);

/* Route (b), materialise G (Eq. 1) then Phi = P_out^T G P_in. */
void oracle_project_materialized(int64_t N, int64_t T, int64_t d_in, int64_t d_out,
                                 int64_t k_in, int64_t k_out, uint64_t seed, uint32_t layer,
                                 int32_t kind, const double* A, const double* B, double* phi);

/* ---- unprojected similarity <DW_q, DW_i>_F ---- */

/* Materialised route: Frobenius inner product of the Eq. 1 matrices.
 * S[q][i] for n_q query and n_t train examples. */
void oracle_similarity_materialized(int64_t T, int64_t d_in, int64_t d_out,
                                    int64_t n_q, const double* Aq, const double* Bq,
                                    int64_t n_t, const double* At, const double* Bt, double* S);
/* Factorised route, Eq. 4: sum_{t,s} <a_t^q, a_s^i> <g_t^q, g_s^i>. */
void oracle_similarity_gram(int64_t T, int64_t d_in, int64_t d_out,
                            int64_t n_q, const double* Aq, const double* Bq,
                            int64_t n_t, const double* At, const double* Bt, double* S);

/* ---- per-example gradient norms (App. A.4: norms are routed like Gram
 *      matrices) and cosine scores ---- */

/* ||DW||_F^2 of each of N examples: materialised (Eq. 1, sum of squares). */
void oracle_sq_norms_materialized(int64_t N, int64_t T, int64_t d_in, int64_t d_out,
                                  const double* A, const double* B, double* out);
/* ||DW||_F^2 by Eq. 4 with both sides the same example:
 * sum_{t,s} <a_t, a_s> <g_t, g_s>. */
void oracle_sq_norms_gram(int64_t N, int64_t T, int64_t d_in, int64_t d_out,
                          const double* A, const double* B, double* out);
/* Cosine scores C[q][i] = S[q][i] / sqrt(nq[q] * nt[i]) from squared norms. */
void oracle_cosine(int64_t n_q, int64_t n_t, const double* S, const double* nq,
                   const double* nt, double* C);

/* ---- curvature preconditioning of the queries (App. B.2, B.3) ---- */

/* F = (1/N) sum_i phi_i phi_i^T (D x D). */
void oracle_fisher(int64_t D, int64_t N, const double* phi, double* F);
/* lambda = lambda_abs + lambda_rel * tr(F)/D (tr(F)/D is the mean eigenvalue). */
double oracle_damping(int64_t D, const double* F, double lambda_abs, double lambda_rel);
/* The same lambda from the N x D features directly (tr(F) = sum_a (1/N) sum_n phi_na^2). */
double oracle_damping_features(int64_t D, int64_t N, const double* phi, double lambda_abs,
                               double lambda_rel);
/* In-place lower Cholesky factor of the D x D SPD matrix M (upper part zeroed).
 * Returns 0, or j+1 if the leading minor of order j+1 is not positive. */
int32_t oracle_cholesky(int64_t D, double* M);
/* Qhat = (F + lambda I)^{-1} Q for n_q row vectors Q[q][:] (D each). */
int32_t oracle_precondition(int64_t D, const double* F, double lambda,
                            int64_t n_q, const double* Q, double* Qhat);
/* The same Qhat = (F + lambda I)^{-1} Q with F = (1/N) Phi^T Phi given by its
 * N x D features, through the Woodbury identity (an N x N solve). */
int32_t oracle_precondition_lowrank(int64_t D, int64_t N, const double* phi, double lambda,
                                    int64_t n_q, const double* Q, double* Qhat);

/* ---- Kronecker-factored curvature on the projected factors (K-FAC of
 *      Martens & Grosse 2015, EK-FAC of George et al. 2018; the paper applies
 *      them to projected factors unchanged, App. A.2, and damps by a multiple
 *      of each layer's mean eigenvalue, App. B.2) ---- */

/* Token-averaged second moments of the projected factors of N examples:
 * Ca = (1/(N T)) sum_i sum_t a~_t a~_t^T (k_in x k_in) and
 * Cg = (1/(N T)) sum_i sum_t g~_t g~_t^T (k_out x k_out), a~_t = P_a a_t,
 * g~_t = P_g g_t with the seeded maps. */
void oracle_kfac_covariances(int64_t N, int64_t T, int64_t d_in, int64_t d_out,
                             int64_t k_in, int64_t k_out, uint64_t seed, uint32_t layer,
                             int32_t kind, const double* A, const double* B,
                             double* Ca, double* Cg);
/* Symmetric eigendecomposition C = U diag(w) U^T by the cyclic Jacobi method
 * (Golub & Van Loan, Matrix Computations, Sec. 8.5): eigenvalues ascending in
 * w, eigenvectors in the columns of U (row-major n x n). Returns the number of
 * sweeps, or -1 if 100 sweeps did not converge. */
int32_t oracle_sym_eig(int64_t n, const double* C, double* w, double* U);
/* K-FAC eigenvalues of Cg (x) Ca in the Kronecker eigenbasis:
 * Lam[r][c] = wg[r] * wa[c] (k_out x k_in). */
void oracle_kfac_eigenvalues(int64_t k_in, int64_t k_out, const double* wa, const double* wg,
                             double* Lam);
/* EK-FAC eigenvalue correction: the mean over the N training features of the
 * squared coordinates in the Kronecker eigenbasis,
 * Lam[r][c] = (1/N) sum_i ((Ug^T Phi_i Ua)[r][c])^2. */
void oracle_ekfac_eigenvalues(int64_t N, int64_t k_in, int64_t k_out, const double* phi,
                              const double* Ua, const double* Ug, double* Lam);
/* lambda = lambda_abs + lambda_rel * mean(Lam). */
double oracle_kfac_damping(int64_t k_in, int64_t k_out, const double* Lam, double lambda_abs,
                           double lambda_rel);
/* Qhat = Ug [(Ug^T Q Ua) / (Lam + lambda)] Ua^T for n_q query features
 * (each k_out x k_in, row-major), the inverse of the damped curvature
 * applied in its eigenbasis. */
void oracle_kfac_precondition(int64_t k_in, int64_t k_out, const double* Ua, const double* Ug,
                              const double* Lam, double lambda, int64_t n_q, const double* Q,
                              double* Qhat);

/* ---- token-level scores and random-mask reduction ---- */

/* Token-level decomposition (appendix on token-level attribution): for train
 * example i and query matrix R_j (k_out x k_in, row-major; e.g. a projected,
 * possibly preconditioned query feature),
 *   s[j][i][t] = g~_t^T R_j a~_t  with a~_t = P_a a_t, g~_t = P_g g_t,
 * so that sum_t s[j][i][t] = <Phi_i, R_j>. out is n_q x N x T. */
void oracle_token_scores(int64_t N, int64_t T, int64_t d_in, int64_t d_out, int64_t k_in,
                         int64_t k_out, uint64_t seed, uint32_t layer, int32_t kind,
                         const double* A, const double* B, int64_t n_q, const double* R,
                         double* out);
/* Random-mask reduction gathered from the factors: for each example and each
 * mask coordinate (rows[m], cols[m]) of DW, the entry
 *   out[n][m] = sum_t g_t[rows[m]] a_t[cols[m]]    (Eq. 1 at that entry). */
void oracle_mask_gather(int64_t N, int64_t T, int64_t d_in, int64_t d_out, const double* A,
                        const double* B, int64_t n_coords, const int32_t* rows,
                        const int32_t* cols, double* out);

/* ---- scores and ranking ---- */

/* S[q][i] = sum_f Qhat[q][f] Phi[i][f]. */
void oracle_score(int64_t n_q, int64_t n_t, int64_t D,
                  const double* Qhat, const double* phi, double* S);
/* Per row of S (n_q x n_t), the k largest entries, descending, ties broken
 * by the smaller train index; NaN ranks above every number, -0 equals +0. */
void oracle_topk(int64_t n_q, int64_t n_t, const double* S, int32_t k,
                 int32_t* idx, double* val);

/* ---- FLOP cost of each route (App. A.4, Table 2) ---- */

/* op 0 = project N=n1 examples; op 1 = n1 x n2 similarity of projected
 * gradients; op 2 = n1 x n2 exact (unprojected) similarity; op 3 = squared
 * norms of n1 projected gradients; op 4 = squared norms of n1 unprojected
 * gradients.
 * cost[0] factored, cost[1] materialised, cost[2] Gram; a route that does not
 * produce the op's result gets -1. Returns the index of the cheapest route
 * (ties go to the lower index, i.e. the factored side). */
int32_t oracle_route_costs(int32_t op, int64_t n1, int64_t n2, int64_t T,
                           int64_t d_in, int64_t d_out, int64_t k_in, int64_t k_out,
                           double cost[3]);

/* Threads the oracle's parallel loops may use (1 = serial). */
void oracle_set_threads(int32_t n);
int32_t oracle_get_threads(void);

#ifdef __cplusplus
}
#endif
#endif /* TDA_ORACLE_H */
