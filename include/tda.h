/*
 * tda.h -- C ABI of the GB300 (sm_103a) training-data-attribution hot path.
 *
 * The library turns per-example weight gradients of linear layers, given in
 * factored form, into seeded Kronecker-projected features, preconditions the
 * queries with a damped Fisher inverse (or K-FAC / EK-FAC on the projected
 * factors) and scores queries against training examples, routing each layer
 * and operation between factored, materialised and Gram forms (dattri-LLM
 * paper, Sec. 3.2 and App. A.2, A.4, B.2, B.3). It also computes routed
 * per-example gradient norms and cosine scores, token-level score
 * decompositions and random-mask reductions from the same factors.
 *
 * Notation. A linear layer z = W a has W in R^{N_o x N_i}. For one example with
 * T token positions the paper's factors are a in R^{N_i x T} and g = Dz in
 * R^{N_o x T}, and the weight gradient is DW = g a^T = sum_t g_t a_t^T
 * (Eq. 1). This ABI stores an example's factors token-major:
 *     A[t][c] = a_t[c]   (T x d_in,  d_in  = N_i)
 *     B[t][r] = g_t[r]   (T x d_out, d_out = N_o)
 * and a batch of N examples as A[N][T][d_in], B[N][T][d_out], C-contiguous.
 * A padded token is a zero row in both A and B; it contributes nothing.
 *
 * Projection (Eq. 2, App. A.2). P_a (k_in x d_in) and P_g (k_out x d_out) are
 * Rademacher maps with entries s/sqrt(k), s in {+1,-1}, k the map's output
 * dimension. s is generated from (seed, layer, side, row, col) by a
 * counter-based hash; the matrices never exist in device memory. A projected
 * feature is the k_out x k_in matrix
 *     Phi = P_g DW P_a^T = (B S_out)^T (A S_in) / sqrt(k_in k_out)
 * stored row-major (feature index i*k_in + j), D = k_in*k_out features.
 *
 * Conventions shared by every entry point:
 *  - All pointers to tensors are DEVICE pointers (cudaMalloc'd, or from a
 *    caching allocator) unless a comment says host. The caller owns every
 *    buffer; the library allocates no device memory. Scratch is passed in as
 *    `ws` of `ws_bytes`, sized by tda_workspace_size().
 *  - `stream` is a cudaStream_t (NULL = legacy default stream). Every call is
 *    asynchronous on that stream unless its comment says otherwise.
 *  - Arguments are validated on the host before any launch; a failing call
 *    launches nothing and returns a non-zero tda_status. tda_last_error()
 *    returns a thread-local message describing the last failure.
 *  - Device-side bounded waits that time out set a device error word instead
 *    of hanging; tda_device_status() synchronises the stream and reports it.
 *  - Nothing throws across the ABI.
 */
#ifndef TDA_H
#define TDA_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
    TDA_OK = 0,
    TDA_ERR_INVALID_ARG = 1, /* null pointer, bad size, misalignment, bad enum */
    TDA_ERR_UNSUPPORTED = 2, /* valid request with no kernel for it (e.g. route) */
    TDA_ERR_WORKSPACE = 3,   /* ws smaller than tda_workspace_size() */
    TDA_ERR_CUDA = 4,        /* a CUDA runtime call failed; see tda_last_error */
    TDA_ERR_NOT_SPD = 5,     /* F + lambda I was not positive definite */
    TDA_ERR_TIMEOUT = 6      /* a device-side bounded wait expired */
} tda_status;

typedef enum { TDA_F32 = 0, TDA_BF16 = 1, TDA_F64 = 2 } tda_dtype;

/* TDA_PROJ_IDENTITY requires k_in == d_in and k_out == d_out and uses P = I
 * (no 1/sqrt(k) scale), so Phi = DW exactly: the unprojected gradient. */
typedef enum { TDA_PROJ_RADEMACHER = 0, TDA_PROJ_IDENTITY = 1 } tda_proj_kind;

/* Routes (Sec. 3.2 "FLOP-aware routing", App. A.4):
 *  FACTORED    -- project the factors, then contract over tokens (Eq. 2);
 *  MATERIALIZE -- form DW = g a^T (Eq. 1), then project it / dot it;
 *  GRAM        -- factored inner products, sum_{t,s} <a_t,a_s><g_t,g_s> (Eq. 4). */
typedef enum {
    TDA_ROUTE_AUTO = -1,
    TDA_ROUTE_FACTORED = 0,
    TDA_ROUTE_MATERIALIZE = 1,
    TDA_ROUTE_GRAM = 2
} tda_route_id;

/* Operations the cost model routes (App. A.4: per layer and per operation). */
typedef enum {
    TDA_OP_PROJECT = 0,             /* n1 examples -> n1 projected features      */
    TDA_OP_SIMILARITY_PROJECTED = 1,/* n1 x n2 inner products of projected grads */
    TDA_OP_SIMILARITY_EXACT = 2,    /* n1 x n2 inner products of unprojected DW  */
    TDA_OP_NORM_PROJECTED = 3,      /* n1 squared norms of projected gradients   */
    TDA_OP_NORM_EXACT = 4           /* n1 squared norms of unprojected DW        */
} tda_op;

/* One linear layer. seed and layer must be identical for every gradient that
 * will be compared (App. A.2: the per-layer base seed is held fixed). */
typedef struct {
    int64_t d_in;   /* N_i, input width  */
    int64_t d_out;  /* N_o, output width */
    int64_t T;      /* token positions per example */
    int32_t k_in;   /* k_a, projected input dimension  */
    int32_t k_out;  /* k_g, projected output dimension */
    uint64_t seed;  /* base seed of the projection */
    uint32_t layer; /* layer index mixed into the seed */
    int32_t kind;   /* tda_proj_kind */
} tda_layer_desc;

/* ---------------------------------------------------------------------------
 * tda_proj_entries -- write the sign matrix S (rows x cols, int8 in {+1,-1},
 * or {0,1} for the identity kind) of one projection side, exactly as the
 * projection kernels generate it on chip. side 0 = input factor a (S_in,
 * rows = d_in, cols = k_in); side 1 = output gradient g (S_out, rows = d_out,
 * cols = k_out). P = S / sqrt(cols). Seeds per layer and side: App. A.2.
 * out: device, rows*cols bytes, row-major. cols in [1, 1024].
 * ------------------------------------------------------------------------- */
tda_status tda_proj_entries(uint64_t seed, uint32_t layer, int32_t side, int32_t kind,
                            int64_t rows, int32_t cols, int8_t* out, void* stream);

/* ---------------------------------------------------------------------------
 * tda_workspace_size -- bytes of scratch `ws` that the matching call needs
 * (op PROJECT -> tda_project; SIMILARITY_PROJECTED -> tda_similarity_projected;
 * SIMILARITY_EXACT -> tda_similarity_exact; NORM_* -> tda_norms), for one
 * train example per chunk.
 * n1 = examples (or queries), n2 = train examples (similarity only).
 * route AUTO resolves through tda_route() first. Host only; no device work.
 * ------------------------------------------------------------------------- */
tda_status tda_workspace_size(tda_op op, const tda_layer_desc* L, tda_dtype dtype,
                              int64_t n1, int64_t n2, tda_route_id route, size_t* bytes);

/* ---------------------------------------------------------------------------
 * tda_project -- projected per-example gradients of one layer (Eq. 1, Eq. 2).
 *   dtype  TDA_BF16 or TDA_F32: element type of A and B. Accumulation is fp32.
 *   A      device, A[N][T][d_in], 16-byte aligned.
 *   B      device, B[N][T][d_out], 16-byte aligned.
 *   phi    device fp32, N rows of D = k_in*k_out features, row n at
 *          phi + n*ld_phi (ld_phi >= D); overwritten.
 *   route  FACTORED (Eq. 2 on the factors), MATERIALIZE (DW first), or AUTO
 *          (tda_route's choice for TDA_OP_PROJECT).
 * Both routes give the same result up to rounding (App. A.4).
 * bf16 requires d_in % 8 == 0 and d_out % 8 == 0; fp32 requires % 4.
 *   ws     MATERIALIZE: required (tda_workspace_size bytes per example in a
 *          chunk). FACTORED on the tensor cores: optional, 256-byte aligned;
 *          with tda_workspace_size bytes the kernel gives every SM an equal
 *          run of 128-token tiles (an example split between SMs is summed in
 *          a fixed order, so results do not depend on timing) and, for
 *          k = 128, reads sign tables written once per call; without it each
 *          SM takes whole examples. Calls that share a ws must not overlap.
 * ------------------------------------------------------------------------- */
tda_status tda_project(const tda_layer_desc* L, tda_dtype dtype, const void* A, const void* B,
                       int64_t N, float* phi, int64_t ld_phi, tda_route_id route,
                       void* ws, size_t ws_bytes, void* stream);

/* Which kernel tda_project (route FACTORED) would run for these arguments on
 * the current device: 1 = the tcgen05/TMA tensor-core kernel (bf16, k_in ==
 * k_out in {16, 32, 64, 128}, sm_103), 0 = the CUDA-core kernel, negative = the
 * arguments are invalid. Host only; for tests and benchmark reports. */
int32_t tda_project_engine(const tda_layer_desc* L, tda_dtype dtype, const void* A, const void* B);

/* ---------------------------------------------------------------------------
 * tda_project_host -- tda_project (route FACTORED) for factors held in HOST
 * memory. A_h[N][T][d_in] and B_h[N][T][d_out] are copied chunk by chunk into
 * two halves of the device scratch `ws` on a copy stream owned by the library
 * and projected on `stream` as they land (App. A.2: factors are projected as
 * they arrive and never buffered whole). Page-locked host memory
 * (cudaHostAlloc / cudaHostRegister) lets copies overlap compute; pageable
 * memory works but serialises. The host buffers must stay unchanged until
 * `stream` has completed. ws: >= tda_project_host_ws_min() bytes (one example
 * per half), 256-byte aligned; larger ws means larger chunks. With at least
 * 2 x tda_workspace_size(TDA_OP_PROJECT, FACTORED) bytes beyond the minimum, the
 * end of ws also serves as the projection's optional workspace (one per half).
 * Calls on one device serialise their enqueueing on a library mutex.
 * ------------------------------------------------------------------------- */
size_t tda_project_host_ws_min(const tda_layer_desc* L, tda_dtype dtype);
tda_status tda_project_host(const tda_layer_desc* L, tda_dtype dtype, const void* A_h, const void* B_h,
                            int64_t N, float* phi, int64_t ld_phi, void* ws, size_t ws_bytes,
                            void* stream);

/* ---------------------------------------------------------------------------
 * tda_project_materialized_noalloc -- tda_project with route MATERIALIZE for
 * callers that cannot allocate device memory: the library keeps its own
 * scratch in a fixed device array of tda_noalloc_scratch_bytes() bytes
 * (64 MiB), held on every GPU that loads libtda.so until the process exits.
 * (The paper has no counterpart; this is a deployment convenience.)
 * Intended for code that cannot call cudaMalloc or supply a workspace where it
 * projects, e.g. a plugin inside a host program that owns all device memory,
 * or a loop that must not pay cudaMalloc's implicit device synchronisation.
 *   Arguments as tda_project; A, B, phi are still the caller's buffers.
 *   Rejects (TDA_ERR_WORKSPACE) a layer whose per-example scratch,
 *   4*(d_out*d_in + d_out*k_in) bytes, exceeds the array.
 *   The first call in a CUDA context (normally the runtime's primary context
 *   of the current device) resolves the array's device address
 *   (cudaGetSymbolAddress) and caches it for that context. Under lazy module
 *   loading (CUDA_MODULE_LOADING=LAZY, the default) that first call is also
 *   when the driver loads the module and commits the 64 MiB, so it can fail
 *   with TDA_ERR_CUDA if the device is full: make the first call at
 *   initialisation, before the host program takes the rest of the memory and
 *   before any stream capture.
 *   Every call shares the one array and leaves its contents behind; the
 *   kernels overwrite what they read, so nothing needs clearing. Calls whose
 *   work overlaps on the GPU (different streams, or host threads without
 *   ordering) race on the array: serialise them on one stream.
 *   No cudaMalloc, cudaFree or allocating library routine is called.
 * ------------------------------------------------------------------------- */
size_t tda_noalloc_scratch_bytes(void);
tda_status tda_project_materialized_noalloc(const tda_layer_desc* L, tda_dtype dtype, const void* A,
                                            const void* B, int64_t N, float* phi, int64_t ld_phi,
                                            void* stream);

/* ---------------------------------------------------------------------------
 * tda_similarity_exact -- unprojected gradient inner products
 *   S[q][i] = beta*S[q][i] + <DW_q, DW_i>_F
 * for n_q query and n_t train examples of one layer (Eq. 4's left side).
 *   route GRAM computes sum_{t,s} <a_t^q,a_s^i><g_t^q,g_s^i> (Eq. 4) without
 *   forming DW; MATERIALIZE forms DW (Eq. 1) in ws and takes Frobenius dots
 *   split over slices of the d_out*d_in features (ws also holds the slices'
 *   partial sums; a larger ws holds more train DW at once); AUTO asks tda_route
 *   (TDA_OP_SIMILARITY_EXACT).
 *   Aq/Bq: [n_q][T][d], At/Bt: [n_t][T][d], dtype as in tda_project.
 *   S: device fp32, row q at S + q*ld_S (ld_S >= n_t). beta 0 overwrites.
 * ------------------------------------------------------------------------- */
tda_status tda_similarity_exact(const tda_layer_desc* L, tda_dtype dtype,
                                const void* Aq, const void* Bq, int64_t n_q,
                                const void* At, const void* Bt, int64_t n_t,
                                float* S, int64_t ld_S, float beta, tda_route_id route,
                                void* ws, size_t ws_bytes, void* stream);

/* Which kernel the GRAM route of tda_similarity_exact runs: 1 = the tcgen05
 * kernel (bf16 factors, T a power of two, d_in and d_out multiples of 8,
 * 16-byte aligned factors, sm_103), whose two token Grams (A_q A_i^T, B_q B_i^T)
 * are tensor-core GEMMs with fp32 accumulation; 0 = the CUDA-core kernel.
 * Host only. */
int32_t tda_similarity_gram_engine(const tda_layer_desc* L, tda_dtype dtype, const void* Aq, const void* Bq,
                                   const void* At, const void* Bt);

/* ---------------------------------------------------------------------------
 * tda_similarity_projected -- inner products of PROJECTED gradients,
 *   S[q][i] = beta*S[q][i] + <Phi_q, Phi_i>,  Phi = P_g DW P_a^T (Eq. 2),
 * by any of the three routes that give this result (App. A.4: routing per
 * operation; exact arithmetic gives the same S):
 *   FACTORED    project both sides' factors (Eq. 2), then dot the features;
 *   MATERIALIZE form DW (Eq. 1), project it, then dot the features;
 *   GRAM        project the factors per token (a~_t = P_a a_t, g~_t = P_g g_t)
 *               and apply Eq. 4 to them, never forming Phi;
 *   AUTO        tda_route(TDA_OP_SIMILARITY_PROJECTED).
 * Arguments as tda_similarity_exact. ws: >= tda_workspace_size(
 * TDA_OP_SIMILARITY_PROJECTED, L, dtype, n_q, n_t, route) bytes, 256-byte
 * aligned; more ws lets train examples go through in larger chunks.
 * ------------------------------------------------------------------------- */
tda_status tda_similarity_projected(const tda_layer_desc* L, tda_dtype dtype,
                                    const void* Aq, const void* Bq, int64_t n_q,
                                    const void* At, const void* Bt, int64_t n_t,
                                    float* S, int64_t ld_S, float beta, tda_route_id route,
                                    void* ws, size_t ws_bytes, void* stream);

/* ---------------------------------------------------------------------------
 * tda_norms -- squared Frobenius norms of per-example gradients, routed like
 * the cross-Gram matrices (App. A.4: "for cross-Gram matrices and for
 * per-example norms alike"); with tda_cosine they give LESS-style cosine
 * scores. op TDA_OP_NORM_PROJECTED: ||Phi_i||^2 of the projected gradient
 * (routes FACTORED, MATERIALIZE, GRAM on projected factors); op
 * TDA_OP_NORM_EXACT: ||DW_i||_F^2 (routes MATERIALIZE, GRAM by Eq. 4 with
 * both sides example i). AUTO asks tda_route. out: device fp32[N].
 * ws >= tda_workspace_size(op, L, dtype, N, 0, route) (0 for exact GRAM).
 * ------------------------------------------------------------------------- */
tda_status tda_norms(tda_op op, const tda_layer_desc* L, tda_dtype dtype, const void* A, const void* B,
                     int64_t N, float* out, tda_route_id route, void* ws, size_t ws_bytes, void* stream);

/* tda_cosine -- S[q][i] <- S[q][i] / sqrt(nq[q] * nt[i]) in place, nq and nt
 * squared norms (device fp32, e.g. from tda_norms); IEEE division semantics
 * (a zero norm gives inf or NaN, visibly). */
tda_status tda_cosine(float* S, int64_t n_q, int64_t n_t, int64_t ld_S, const float* nq, const float* nt,
                      void* stream);

/* ---------------------------------------------------------------------------
 * tda_precondition -- damped Fisher inverse on the query side (App. B.3: a
 * curvature fit over the training gradients, then per-layer preconditioning
 * of the queries; App. B.2: damping in units of the mean eigenvalue), for
 * n_layers independent layers of D features each in one call.
 *
 * Feature layout: layer l's D features of example (or query) row r are at
 * phi[r*ld_phi + l*D + f], q[r*ld_q + l*D + f], qhat[r*ld_qhat + l*D + f]:
 * the layers' features side by side in each row (n_layers = 1: one layer).
 *
 * `state` is a device buffer of n_layers * tda_precondition_state_bytes(D,
 * state_dtype) bytes, 16-byte aligned: per layer a 64-byte header, the D x D
 * matrix M and the inverses of M's 32 x 32 diagonal blocks, all in
 * state_dtype (TDA_F32 or TDA_F64). A job whose training features are sharded
 * over ranks adds the layers' M (bytes [64, 64 + D*D*sizeof) of each layer's
 * state) over the ranks (an all-reduce) between FIT_ACCUM and FACTOR, and
 * passes the global n_total to FACTOR. The ops, in order of use:
 *   TDA_PC_RESET      zero the state.
 *   TDA_PC_FIT_ACCUM  M_l += Phi_l^T Phi_l over n feature rows. Call once per
 *                     streamed chunk of training features. Only the lower
 *                     triangle (column <= row) of M_l is guaranteed (FACTOR
 *                     reads nothing else); an F32 state accumulates in fp32
 *                     from 3xTF32 tensor-core products for D >= 128.
 *   TDA_PC_FACTOR     F_l = M_l / n_total; lambda_l = lambda_abs +
 *                     lambda_rel_mean_eig * tr(F_l)/D; factor F_l + lambda_l I
 *                     = L L^T (Cholesky) into the state. A non-positive pivot
 *                     is recorded in the layer's header; tda_precondition_info
 *                     reports it (TDA_ERR_NOT_SPD).
 *   TDA_PC_APPLY      qhat_l = (F_l + lambda_l I)^{-1} q_l for n_q query rows
 *                     (q fp32; qhat in state_dtype, i.e. fp64 rows for an F64
 *                     state). Layers whose FACTOR failed get NaN rows.
 *                     Needs D <= 40960 (F32) or 20480 (F64).
 *   TDA_PC_FACTOR_APPLY  FACTOR, then APPLY, in one call (same arguments and
 *                     results as the two; a failed layer's rows are NaN). For an
 *                     F32 state with D a multiple of 32 below 2048 and n_q <= 256
 *                     both run in one launch: the query rows are solved alongside
 *                     the factorisation (forward substitution as extra rows of
 *                     each step) and then backward. qhat may not alias q.
 * Large layers (F32 state, D a multiple of 128, D >= 2048): FACTOR is a blocked
 * Cholesky in 256-column panels whose trailing updates run on the tensor cores
 * (3xTF32, fp32-accurate); it also leaves L^T in M's upper triangle, and APPLY
 * (qhat 16-byte aligned, ld_qhat a multiple of 4) then solves the query rows in
 * 128-column blocks with tensor-core updates. In this mode qhat may alias q
 * (same pointer and row stride: solved in place).
 * Arguments not used by an op are ignored (may be 0/NULL).
 * ------------------------------------------------------------------------- */
#define TDA_PC_RESET 0
#define TDA_PC_FIT_ACCUM 1
#define TDA_PC_FACTOR 2
#define TDA_PC_APPLY 3
#define TDA_PC_FACTOR_APPLY 4

/* Bytes of ONE layer's state (a multiple of 256). */
size_t tda_precondition_state_bytes(int64_t D, tda_dtype state_dtype);

tda_status tda_precondition(int32_t op, int32_t n_layers, int64_t D, tda_dtype state_dtype, void* state,
                            const float* phi, int64_t n, int64_t ld_phi,
                            int64_t n_total, double lambda_abs, double lambda_rel_mean_eig,
                            const float* q, int64_t n_q, int64_t ld_q,
                            void* qhat, int64_t ld_qhat, void* stream);

/* Synchronises `stream` and copies each layer's header to host
 * info[4*l .. 4*l+3] = {lambda used, tr(F)/D, failed pivot (0 = SPD), n_total}
 * (info holds 4*n_layers doubles). Returns TDA_ERR_NOT_SPD if the last FACTOR
 * failed for any layer. */
tda_status tda_precondition_info(int32_t n_layers, int64_t D, tda_dtype state_dtype, const void* state,
                                 double* info, void* stream);

/* ---------------------------------------------------------------------------
 * K-FAC and EK-FAC on the projected factors. The paper runs both
 * Kronecker-factored curvature methods (Martens & Grosse 2015; George et al.
 * 2018) on the projected pair (a~_t, g~_t) unchanged (App. A.2) and damps
 * each layer by a multiple of its mean eigenvalue (App. B.2, 0.1 for EK-FAC).
 * Per layer, with a~_t = P_a a_t (k_in) and g~_t = P_g g_t (k_out):
 *   C_a = (1/M) sum a~_t a~_t^T,  C_g = (1/M) sum g~_t g~_t^T  (M = N*T token
 *   positions of the N training examples seen),
 *   C_a = U_a diag(alpha) U_a^T, C_g = U_g diag(gamma) U_g^T,
 *   K-FAC eigenvalues  Lam[r][c] = gamma_r alpha_c,
 *   EK-FAC eigenvalues Lam[r][c] = (1/N) sum_i ((U_g^T Phi_i U_a)[r][c])^2,
 *   lambda = lambda_abs + lambda_rel * mean(Lam),
 *   Qhat = U_g [(U_g^T Q U_a) / (Lam + lambda)] U_a^T  per query feature
 *   (Q, Qhat, Phi: k_out x k_in row-major, index r*k_in + c, as tda_project).
 *
 * `state`: device buffer of n_layers * tda_kfac_state_bytes(k_in, k_out) bytes
 * (layer l at byte l * tda_kfac_state_bytes), 16-byte aligned, fp64 per layer:
 * an 8-double header (M, N, Jacobi sweeps), the factor sums, the eigenbases and
 * eigenvalues, the EK-FAC sums. The sums, in doubles from the layer's start
 * (ka = k_in, kg = k_out): [0] M; [8, 8 + ka^2) sum a~a~^T; [8 + ka^2,
 * 8 + ka^2 + kg^2) sum g~g~^T; [1] N and [Le, Le + ka*kg) the EK-FAC sums, with
 * Le = 8 + 2 ka^2 + 2 kg^2 + ka + kg. A job whose training examples are
 * sharded over ranks adds these ranges over the ranks (an all-reduce) before
 * tda_kfac_eigen, respectively before tda_kfac_apply for EK-FAC. The n_layers calls (reset, eigen,
 * accumulate_eigenvalues, apply) treat that many layers of equal k_in, k_out in
 * one launch, their features side by side in each row (layer l at column
 * l*k_in*k_out, as tda_precondition); accumulate_factors and project_kfac take
 * one layer's factors and that layer's state. Calls in order of use:
 *   tda_kfac_reset                 zero the state.
 *   tda_kfac_accumulate_factors    add the factor covariance sums of N training
 *                                  examples (A, B as tda_project). ws >=
 *                                  tda_kfac_workspace_size(L, dtype). Call once
 *                                  per streamed chunk.
 *   tda_project_kfac               tda_project (factored route) that also adds
 *                                  the factor covariance sums, in one pass over
 *                                  the factors (bf16, the tensor-core kernel's
 *                                  shapes; TDA_ERR_UNSUPPORTED otherwise).
 *   tda_kfac_eigen                 C = sums / M; both eigendecompositions
 *                                  (parallel cyclic Jacobi: for k <= 64 fp32
 *                                  sweeps, then the fp32 eigenvectors made
 *                                  orthonormal in fp64 and fp64 sweeps on
 *                                  V^T C V; fp64 sweeps throughout for larger k;
 *                                  at most 60 fp64 sweeps, their count, or -1 if
 *                                  they did not converge, lands in header[2] (a)
 *                                  and [3] (g)). Resets the EK-FAC sums.
 *   tda_kfac_accumulate_eigenvalues  EK-FAC: add sum_i (U_g^T Phi_i U_a)^2 over n
 *                                  training features (rows of stride ld_phi).
 * ws (device scratch, 256-byte aligned) of tda_kfac_workspace_size(L, dtype)
 * bytes serves every call that takes one; more lets accumulate_factors
 * process more examples per pass.
 *   tda_kfac_apply                 Qhat for n_q query rows; kind TDA_KFAC or
 *                                  TDA_EKFAC.
 * Supports 1 <= k_in, k_out <= 128. Errors: TDA_ERR_INVALID_ARG for bad sizes
 * or pointers, TDA_ERR_WORKSPACE for a short ws.
 * ------------------------------------------------------------------------- */
#define TDA_KFAC 0
#define TDA_EKFAC 1
size_t tda_kfac_state_bytes(int32_t k_in, int32_t k_out);
size_t tda_kfac_workspace_size(const tda_layer_desc* L, tda_dtype dtype);
tda_status tda_kfac_reset(int32_t n_layers, int32_t k_in, int32_t k_out, void* state, void* stream);
tda_status tda_kfac_accumulate_factors(const tda_layer_desc* L, tda_dtype dtype, const void* A, const void* B,
                                       int64_t N, void* state, void* ws, size_t ws_bytes, void* stream);
tda_status tda_project_kfac(const tda_layer_desc* L, tda_dtype dtype, const void* A, const void* B, int64_t N,
                            float* phi, int64_t ld_phi, void* state, void* ws, size_t ws_bytes, void* stream);
tda_status tda_kfac_eigen(int32_t n_layers, int32_t k_in, int32_t k_out, void* state, void* stream);
tda_status tda_kfac_accumulate_eigenvalues(int32_t n_layers, int32_t k_in, int32_t k_out, void* state,
                                           const float* phi, int64_t n, int64_t ld_phi, void* ws, size_t ws_bytes,
                                           void* stream);
tda_status tda_kfac_apply(int32_t kind, int32_t n_layers, int32_t k_in, int32_t k_out, const void* state,
                          double lambda_abs, double lambda_rel, const float* q, int64_t n_q, int64_t ld_q,
                          float* qhat, int64_t ld_qhat, void* stream);

/* ---------------------------------------------------------------------------
 * tda_token_scores -- token-level decomposition of the score (token-level
 * attribution appendix): for query matrix R_j and train example i,
 *   out[j*ld_q_out + i*T + t] = beta*out + g~_t^T R_j a~_t,
 * with a~_t = P_a a_t, g~_t = P_g g_t the projected factors of token t of
 * example i (identity kind: the raw factors, R_j then a full d_out x d_in
 * matrix); sum_t of the result is <Phi_i, R_j>. Summing layers: call per
 * layer with beta 1.
 *   A, B   [N][T][d] (dtype as tda_project), device.
 *   R      n_q rows of k_out*k_in fp32 (row-major [k_out][k_in], e.g. a
 *          layer's columns of the preconditioned queries), row stride ld_R.
 *   out    device fp32, ld_q_out >= N*T.
 *   ws     >= tda_token_scores_workspace_size(L) bytes (one example's
 *          projected factors; more lets a pass cover more examples).
 * k_in, k_out <= 128.
 * ------------------------------------------------------------------------- */
size_t tda_token_scores_workspace_size(const tda_layer_desc* L);
tda_status tda_token_scores(const tda_layer_desc* L, tda_dtype dtype, const void* A, const void* B, int64_t N,
                            const float* R, int64_t n_q, int64_t ld_R, float* out, int64_t ld_q_out, float beta,
                            void* ws, size_t ws_bytes, void* stream);

/* ---------------------------------------------------------------------------
 * tda_mask_gather -- random-mask reduction gathered from the factors (the
 * reduced representation of App. B.4: a set of DW coordinates per layer,
 * e.g. ten disjoint masks of 512 or 8192 entries):
 *   out[n*ld_out + m] = sum_t g_t[rows[m]] a_t[cols[m]]  (Eq. 1 at that entry)
 * for each of N examples and n_coords coordinates, without forming DW.
 *   rows, cols  device int32 [n_coords] (the caller draws the masks); a
 *               coordinate outside [0, d_out) x [0, d_in) yields NaN.
 *   out         device fp32, ld_out >= n_coords.
 * Scores of disjoint masks averaged = one tda_score over the concatenated
 * coordinates divided by the mask count. Needs d_in, d_out <= 65536 and
 * (d_in + d_out) * sizeof(dtype) <= 48 KiB.
 * ------------------------------------------------------------------------- */
tda_status tda_mask_gather(const tda_layer_desc* L, tda_dtype dtype, const void* A, const void* B, int64_t N,
                           const int32_t* rows, const int32_t* cols, int64_t n_coords, float* out, int64_t ld_out,
                           void* stream);

/* ---------------------------------------------------------------------------
 * tda_score -- S[q][i] = beta*S[q][i] + sum_f Qhat[q][f] Phi[i][f]
 * (gradient inner products; GradDot when Qhat = Q, Sec. 3.2 / Eq. 4).
 *   Qhat  device, n_q rows of D, q_dtype TDA_F32 or TDA_F64, row stride ld_q.
 *         With TDA_F64 the sum is accumulated in fp64 (CUDA cores). With
 *         TDA_F32 on sm_103 (aligned rows, D >= 64) the sum runs on the tensor
 *         cores as three TF32 products per element pair (hi*hi + hi*lo + lo*hi
 *         of the split x = hi + lo), accurate to about fp32 rounding at the
 *         feature counts of a block (1e-5 relative at D = 7168). The tensor
 *         pipe's fp32 accumulators add with truncation, so the error grows with
 *         the features per call: rows of ~10^6 features are better scored in
 *         blocks of features accumulated with beta = 1.
 *   Phi   device fp32, n_t rows of D, row stride ld_phi.
 *   S     device fp32, row stride ld_S >= n_t. beta 0 overwrites (S may hold
 *         garbage); beta 1 accumulates layers.
 * ------------------------------------------------------------------------- */
tda_status tda_score(const void* Qhat, tda_dtype q_dtype, int64_t n_q, int64_t ld_q,
                     const float* Phi, int64_t n_t, int64_t ld_phi, int64_t D,
                     float* S, int64_t ld_S, float beta, void* stream);

/* Which kernel tda_score would run: 1 = tcgen05 3xTF32 GEMM (fp32 Qhat,
 * 16-byte aligned rows, D >= 64, sm_103), 0 = the CUDA-core kernel. Host only. */
int32_t tda_score_engine(const void* Qhat, tda_dtype q_dtype, int64_t n_q, int64_t ld_q, const float* Phi,
                         int64_t n_t, int64_t ld_phi, int64_t D);

/* ---------------------------------------------------------------------------
 * tda_topk -- per query row of S (n_q x n_t, fp32, row stride ld_S), the k
 * largest scores in descending order; ties go to the smaller train index.
 * idx: device int32 [n_q][k]; val: device fp32 [n_q][k] (may be NULL).
 * 1 <= k <= min(n_t, 1024). A NaN score is treated as larger than +inf (it
 * ranks first), so it is visible in the output.
 * ------------------------------------------------------------------------- */
tda_status tda_topk(const float* S, int64_t n_q, int64_t n_t, int64_t ld_S, int32_t k,
                    int32_t* idx, float* val, void* stream);

/* ---------------------------------------------------------------------------
 * tda_route -- the FLOP-aware route choice (Sec. 3.2, App. A.4, Table 2).
 * Host only, no device work. cost_out[r] = estimated cost of route r
 * (FACTORED, MATERIALIZE, GRAM); -1 for a route that cannot produce the op's
 * result. In the default model the cost is the route's flop count (2 flops
 * per multiply-add); after tda_route_calibrate() it is the estimated seconds
 * max(flops / rate_r, bytes_r / bandwidth) with rates measured on the device.
 * The cheapest route wins; ties prefer GRAM, then FACTORED, then MATERIALIZE.
 * ------------------------------------------------------------------------- */
tda_status tda_route(const tda_layer_desc* L, tda_op op, int64_t n1, int64_t n2,
                     tda_dtype dtype, tda_route_id* chosen, double* cost_out);

/* Measures per-route throughput on the current device with short synthetic
 * launches of the route kernels inside the caller's scratch `ws` (at least
 * TDA_CALIBRATE_WS_BYTES bytes, contents destroyed), synchronises `stream`,
 * then switches tda_route to the time model. rates_out (host, may be NULL)
 * receives 7 doubles: flop/s of [0] the factored projection, [1] building DW
 * (materialise route; tensor cores for bf16 on sm_103), [2] the Gram route on
 * bf16 factors (exact similarity; tensor cores), [3] the Gram route on fp32
 * factors (projected factors, fp32 layers, norms), [4] projecting a built DW
 * with the signs, [5] Frobenius inner products of built DWs; [6] the streaming
 * bytes/s of the factored kernel. The materialise route's time is its DW
 * construction at [1] plus the rest at [4] or [5]. Rates are measured on bf16
 * factors. */
#define TDA_CALIBRATE_WS_BYTES ((size_t)768 << 20)
tda_status tda_route_calibrate(void* ws, size_t ws_bytes, void* stream, double* rates_out);
/* 0 = flop model (the paper's), 1 = calibrated time model. */
tda_status tda_route_set_model(int32_t model);

/* Self-test of the failure path: launches one thread that waits on an
 * mbarrier nothing arrives on, bounded by timeout_ns (at most 2 s) of
 * %globaltimer, exactly like the tensor-core kernels' waits. The wait runs
 * out, the kernel records the timeout and returns; the next
 * tda_device_status() reports TDA_ERR_TIMEOUT and the context stays usable. */
tda_status tda_selftest_bounded_wait(uint64_t timeout_ns, void* stream);

/* Synchronises `stream`, then reads and clears the device error word.
 * Returns TDA_ERR_TIMEOUT if a kernel's bounded wait expired since the last
 * check, TDA_ERR_CUDA on a CUDA error, else TDA_OK. */
tda_status tda_device_status(void* stream);

/* Thread-local message of the last failing call on this thread ("" if none). */
const char* tda_last_error(void);

/* ABI version: major*10000 + minor*100 + patch. */
int32_t tda_version(void);

/* Number of kernel launches this library has issued in this process (all
 * devices, all threads). Host only; for counting launches in a timed region. */
uint64_t tda_launch_count(void);

/* SM budget of the tensor-core factored projection (no counterpart in the
 * paper, which runs PyTorch ops on one stream). That kernel is persistent,
 * one CTA per SM; with n_sms > 0 its later launches use at most n_sms CTAs so
 * that kernels queued on another stream (the query side of a step: the query
 * projection, the curvature fit, its factorisation and the preconditioning)
 * find SMs free and run beside it. 0 (the default) = every SM. Process-wide,
 * host only; results do not depend on it. n_sms < 0 -> TDA_ERR_INVALID_ARG. */
tda_status tda_set_sm_budget(int32_t n_sms);
int32_t tda_get_sm_budget(void);

#ifdef __cplusplus
}
#endif
#endif /* TDA_H */
