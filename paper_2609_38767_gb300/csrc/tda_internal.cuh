// tda_internal.cuh -- internal declarations shared by the CUDA translation
// units of libtda.so (kernels and the C-ABI layer). Not installed.
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

#include <atomic>

#include "../../include/tda.h"

namespace tda {

// ---------------------------------------------------------------------------
// Counter-based Rademacher signs (App. A.2: Rademacher maps, two sides with
// distinct seeds derived from one per-layer base seed).
//
// side_key(seed, layer, side) = mix(mix(seed + G*(layer+1)) + G*(side+1))
// entry (r, c) of a side's d x k sign matrix = bit (r mod 64) of
//   mix(side_key + G*(((c << 32) | (r >> 6)) + 1)),  set bit -> -1.
// mix is the SplitMix64 output function. One 64-bit word therefore holds the
// signs of 64 consecutive rows of one column: exactly one 128-byte row of a
// K-major bf16 operand tile with a 64-wide K chunk.
// ---------------------------------------------------------------------------
constexpr uint64_t kGamma = 0x9E3779B97F4A7C15ull;

__host__ __device__ __forceinline__ uint64_t mix64(uint64_t z) {
    z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
    z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
    return z ^ (z >> 31);
}

__host__ __device__ __forceinline__ uint64_t side_key(uint64_t seed, uint32_t layer, int side) {
    uint64_t base = mix64(seed + kGamma * ((uint64_t)layer + 1u));
    return mix64(base + kGamma * ((uint64_t)(uint32_t)side + 1u));
}

// Sign word of column c for rows [64*rb, 64*rb + 64).
__host__ __device__ __forceinline__ uint64_t sign_word(uint64_t key, uint32_t c, uint64_t rb) {
    return mix64(key + kGamma * ((((uint64_t)c << 32) | rb) + 1u));
}

// Error bits written by kernels into the device error word.
enum : unsigned int {
    kErrTimeout = 1u,    // a bounded mbarrier / flag wait expired
    kErrBadLaunch = 2u,  // a kernel found its launch geometry inconsistent
};

// 1/sqrt(k_in k_out) for Rademacher maps, 1 for the identity map (App. A.2).
float projection_scale(const tda_layer_desc& L);

// Host-side count of kernels this library has launched (tda_launch_count).
void note_launches(uint64_t n);
// tda_set_sm_budget's cap on the persistent projection grid (0 = none).
int sm_budget();

// Device address of the library's error word on the current device.
unsigned int* device_error_word();

// Thread-local error message helpers (api.cu).
tda_status fail(tda_status st, const char* fmt, ...);
tda_status cuda_check(cudaError_t e, const char* what);

// ---------------------------------------------------------------------------
// Kernel launchers (one per translation unit). All return cudaError_t from
// cudaGetLastError() after the launch; arguments are validated by the caller.
// ---------------------------------------------------------------------------

cudaError_t launch_proj_entries(uint64_t key, int kind, int64_t rows, int32_t cols, int8_t* out,
                                cudaStream_t s);

// Generic (SIMT) projection, any shape, fp32 or bf16 inputs.
cudaError_t launch_project_simt(const tda_layer_desc& L, tda_dtype dt, const void* A, const void* B,
                                int64_t N, float* phi, int64_t ld_phi, cudaStream_t s);

// tcgen05 / TMA projection for bf16 inputs. Returns cudaErrorNotSupported if
// the shape has no tensor-core instantiation (caller falls back to SIMT).
bool project_tc_supported(const tda_layer_desc& L, const void* A, const void* B);
bool project_tc_plain_supported(const tda_layer_desc& L, const void* A, const void* B);  // also k = 128
cudaError_t launch_project_tc_kfac(const tda_layer_desc& L, const void* A, const void* B, int64_t N, float* phi,
                                   int64_t ld_phi, float* cov, int* grid_out, unsigned int* err, cudaStream_t s);
int project_tc_max_grid();
cudaError_t launch_project_factors_tc(const tda_layer_desc& L, const void* A, const void* B, int64_t N, float* Y,
                                      unsigned int* err, cudaStream_t s);
// K-FAC / EK-FAC (k_kfac.cu)
size_t kfac_state_bytes(int64_t k_in, int64_t k_out);
int kfac_partial_blocks(int64_t rows);
int64_t kfac_offset_sa(int64_t ka, int64_t kg);
int64_t kfac_offset_sg(int64_t ka, int64_t kg);
cudaError_t launch_kfac_cov(const float* Y, int64_t rows, int k, double* S, double scale, double* header,
                            double add_m, float* part, cudaStream_t s);
cudaError_t launch_kfac_sum_partials(const float* part, int nblk, int64_t stride, int64_t n, double* S, double scale,
                                     double* header, int slot, double add, cudaStream_t s);
cudaError_t launch_kfac_eigen(int n_layers, double* state, int64_t ka, int64_t kg, cudaStream_t s);
cudaError_t launch_kfac_ekfac_accum(int n_layers, double* state, int64_t ka, int64_t kg, const float* phi, int64_t n,
                                    int64_t ld, float* part, int nblk, cudaStream_t s);
cudaError_t launch_kfac_apply(int kind, int n_layers, const double* state, int64_t ka, int64_t kg, double lambda_abs,
                              double lambda_rel, const float* q, int64_t n_q, int64_t ld_q, float* qhat,
                              int64_t ld_qhat, cudaStream_t s);
// Token-level scores and random-mask gather (k_tokens.cu)
cudaError_t launch_token_scores(const float* Ya, const float* Yb, int64_t n, int64_t T, int ka, int kg,
                                const float* R, int64_t n_q, int64_t ld_R, float scale, float* out, int64_t ld_q,
                                int64_t i0, float beta, cudaStream_t s);
int mask_gather_tokens_per_pass(int64_t d_in, int64_t d_out, size_t el);
// Token-level scores on tcgen05, 3xTF32 (k_tokens_tc.cu): k_in = 32, k_out in {16, 32, 64};
// Rs is token_tc_split_bytes of scratch for R's hi and lo halves.
size_t token_tc_split_bytes(int ka, int kg, int64_t n_q);
bool token_tc_supported(int ka, int kg, int64_t n_q);
cudaError_t launch_token_scores_tc(const float* Ya, const float* Yb, int64_t n, int64_t T, int ka, int kg,
                                   const float* R, int64_t n_q, int64_t ld_R, float scale, float* out, int64_t ld_q,
                                   int64_t i0, float beta, float* Rs, cudaStream_t s);
cudaError_t launch_mask_gather(const tda_layer_desc& L, tda_dtype dt, const void* A, const void* B, int64_t N,
                               const int32_t* rows, const int32_t* cols, int64_t n_coords, float* out, int64_t ld_out,
                               cudaStream_t s);
// Route (b)'s materialisation on tcgen05 for bf16 factors (k_materialize_tc.cu)
bool materialize_tc_supported(const tda_layer_desc& L, tda_dtype dt, const void* A, const void* B, const float* G);
cudaError_t launch_materialize_tc(const tda_layer_desc& L, const void* A, const void* B, int64_t e0, int64_t n,
                                  float* G, unsigned int* err, cudaStream_t s);
// ws (optional, 256-byte aligned): for k = 128, >= project_tc_sign_table_bytes(L)
// bytes let the kernel read precomputed sign tiles by TMA instead of generating them;
// >= project_tc_ws_bytes(L) bytes also balance token tiles across the SMs (partial
// blocks of examples split between CTAs after the sign tables).
size_t project_tc_sign_table_bytes(const tda_layer_desc& L);
size_t project_tc_ws_bytes(const tda_layer_desc& L);
cudaError_t launch_project_tc(const tda_layer_desc& L, const void* A, const void* B, int64_t N,
                              float* phi, int64_t ld_phi, unsigned int* err, cudaStream_t s,
                              void* ws = nullptr, size_t ws_bytes = 0);

// Route (b): materialise G = B^T A for nb examples into ws, then project it.
size_t materialize_ws_bytes_per_example(const tda_layer_desc& L);
cudaError_t launch_project_materialized(const tda_layer_desc& L, tda_dtype dt, const void* A,
                                        const void* B, int64_t N, float* phi, int64_t ld_phi,
                                        void* ws, size_t ws_bytes, cudaStream_t s);

// Unprojected similarity, routes (b) and (c).
size_t similarity_materialize_ws_bytes(const tda_layer_desc& L, int64_t n_q, int64_t chunk);
cudaError_t launch_similarity_materialized(const tda_layer_desc& L, tda_dtype dt, const void* Aq,
                                           const void* Bq, int64_t n_q, const void* At,
                                           const void* Bt, int64_t n_t, float* S, int64_t ld_S,
                                           float beta, void* ws, size_t ws_bytes, cudaStream_t s);
// Route (c) on tcgen05 for bf16 factors with T a power of two (k_gram_tc.cu).
bool gram_tc_supported(const tda_layer_desc& L, tda_dtype dt, const void* Aq, const void* Bq, const void* At,
                       const void* Bt);
cudaError_t launch_gram_tc(const tda_layer_desc& L, const void* Aq, const void* Bq, int64_t n_q, const void* At,
                           const void* Bt, int64_t n_t, float* S, int64_t ld_S, float beta, float alpha,
                           unsigned int* err, cudaStream_t s);
cudaError_t launch_similarity_gram(const tda_layer_desc& L, tda_dtype dt, const void* Aq,
                                   const void* Bq, int64_t n_q, const void* At, const void* Bt,
                                   int64_t n_t, float* S, int64_t ld_S, float beta, cudaStream_t s);

// Projected factors (a~ = S_in^T a, g~ = S_out^T g per token, unscaled) and the
// Gram identity on them (projected-similarity route c).
size_t project_factors_bytes_per_example(const tda_layer_desc& L);
cudaError_t launch_project_factors(const tda_layer_desc& L, tda_dtype dt, const void* A, const void* B, int64_t e0,
                                   int64_t n, float* Y, cudaStream_t s);
cudaError_t launch_gram_projected(const tda_layer_desc& L, const float* Yq, int64_t n_q, const float* Yt,
                                  int64_t n_t, float* S, int64_t ld_S, float beta, cudaStream_t s);

// Norms and cosine.
cudaError_t launch_materialize_G(const tda_layer_desc& L, tda_dtype dt, const void* A, const void* B, int64_t e0,
                                 int64_t n, float* G, cudaStream_t s);
cudaError_t launch_row_sq_norms(const float* X, int64_t n, int64_t D, int64_t ld, float* out, cudaStream_t s);
cudaError_t launch_cosine(float* S, int64_t n_q, int64_t n_t, int64_t ld_S, const float* nq, const float* nt,
                          cudaStream_t s);
cudaError_t launch_gram_self(const tda_layer_desc& L, tda_dtype dt, const void* A, const void* B, int64_t n,
                             int64_t d_in, int64_t d_out, float alpha, float* out, cudaStream_t s);

// Preconditioner, n_layers layers of D features each (layer l's columns at
// offset l*D of every feature row).
int64_t precondition_apply_max_d(tda_dtype sdt);
cudaError_t launch_pc_fit(int n_layers, int64_t D, tda_dtype sdt, void* state, const float* phi, int64_t n,
                          int64_t ld, cudaStream_t s);
cudaError_t launch_pc_factor(int n_layers, int64_t D, tda_dtype sdt, void* state, int64_t n_total,
                             double lambda_abs, double lambda_rel, cudaStream_t s);
cudaError_t launch_pc_factor_apply(int n_layers, int64_t D, tda_dtype sdt, void* state, int64_t n_total,
                                   double lambda_abs, double lambda_rel, const float* q, int64_t n_q, int64_t ld_q,
                                   void* qhat, int64_t ld_qhat, cudaStream_t s);
cudaError_t launch_pc_apply(int n_layers, int64_t D, tda_dtype sdt, const void* state, const float* q,
                            int64_t n_q, int64_t ld_q, void* qhat, int64_t ld_qhat, cudaStream_t s);

// Scores and ranking.
cudaError_t launch_score(const void* Qhat, tda_dtype qdt, int64_t n_q, int64_t ld_q,
                         const float* Phi, int64_t n_t, int64_t ld_phi, int64_t D, float* S,
                         int64_t ld_S, float beta, cudaStream_t s);
// Fisher fit on tcgen05 (3xTF32) for an fp32 state: M_l += Phi_l^T Phi_l.
bool fit_tc_supported(int n_layers, int64_t D, const float* phi, int64_t n, int64_t ld);
cudaError_t launch_fit_tc(int n_layers, int64_t D, void* state, size_t state_bytes, const float* phi, int64_t n,
                          int64_t ld, unsigned int* err, cudaStream_t s);

// Score on tcgen05 (3xTF32, fp32-accurate) for an fp32 Qhat.
bool score_tc_supported(tda_dtype qdt, const void* Qhat, int64_t n_q, int64_t ld_q, const float* Phi, int64_t n_t,
                        int64_t ld_phi, int64_t D);
cudaError_t launch_score_tc(const float* Qhat, int64_t n_q, int64_t ld_q, const float* Phi, int64_t n_t, int64_t ld_phi,
                            int64_t D, float* S, int64_t ld_S, float beta, unsigned int* err, cudaStream_t s);
int score_tc_tiles(int64_t n_q, int64_t n_t);
bool gemm_tc_available();  // tcgen05 and the tensor-map encoder are usable on this device
// C[n][m] = beta C[n][m] + alpha sum_k A[m][k] B[n][k] on tcgen05 (3xTF32); lower: square
// symmetric update, tiles on or below the diagonal only. Same operand rules as the score.
cudaError_t launch_gemm_nt_tc(const float* A, int64_t n_a, int64_t lda, const float* B, int64_t n_b, int64_t ldb,
                              int64_t K, float* C, int64_t ldc, float alpha, float beta, bool lower,
                              unsigned int* err, cudaStream_t s);
// The same for nz independent problems in one launch (grid z): problem z's A, B start
// a_z_bytes, b_z_bytes (multiples of 16) after the previous one's, its C c_z floats after.
cudaError_t launch_gemm_nt_tc_batched(const float* A, int64_t n_a, int64_t lda, size_t a_z_bytes, const float* B,
                                      int64_t n_b, int64_t ldb, size_t b_z_bytes, int64_t K, float* C, int64_t ldc,
                                      int64_t c_z, int64_t nz, float alpha, float beta, bool lower,
                                      unsigned int* err, cudaStream_t s);
cudaError_t launch_score_tc_slices(const float* Qhat, int64_t n_q, int64_t ld_q, const float* Phi, int64_t n_t,
                                   int64_t ld_phi, int64_t D, int splits, float* part, unsigned int* err,
                                   cudaStream_t s);
// Split-K score for few, very long rows (Frobenius dots of materialised DW):
// score_dots_tc says whether the tensor-core kernel takes these operands;
// score_splitk_splits plans the feature slices for that kernel (tc) or the
// CUDA-core one; launch_score_splitk runs the plan (part: splits * n_q * n_t floats).
bool score_dots_tc(const float* Q, int64_t n_q, int64_t ld_q, const float* Phi, int64_t n_t, int64_t ld_phi,
                   int64_t D);
int score_splitk_splits(int64_t n_q, int64_t n_t, int64_t D, bool tc);
cudaError_t launch_score_splitk(const float* Q, int64_t n_q, int64_t ld_q, const float* Phi, int64_t n_t,
                                int64_t ld_phi, int64_t D, float* S, int64_t ld_S, float beta, int splits,
                                float* part, bool tc, cudaStream_t s);
cudaError_t launch_topk(const float* S, int64_t n_q, int64_t n_t, int64_t ld_S, int32_t k,
                        int32_t* idx, float* val, cudaStream_t s);

// State header layout of the preconditioner (doubles).
enum { kPcLambda = 0, kPcMeanEig = 1, kPcFailedPivot = 2, kPcNTotal = 3, kPcHeaderDoubles = 8 };

// Per-kernel launch set-up that does not change between launches, done once per device
// (a stream job launches hundreds of kernels a step, and the host's time per launch adds up):
// the dynamic shared-memory limit of kernel K, and K's maximum co-resident clusters of cs CTAs.
template <auto Kernel>
cudaError_t smem_attr_once(int bytes) {
    static std::atomic<uint64_t> done{0};  // bit d: set on device d
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    const uint64_t bit = (dev >= 0 && dev < 64) ? (1ull << dev) : 0;
    if (bit && (done.load(std::memory_order_acquire) & bit)) return cudaSuccess;
    e = cudaFuncSetAttribute(Kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes);
    if (e == cudaSuccess && bit) done.fetch_or(bit, std::memory_order_release);
    return e;
}

template <auto Kernel>
int max_clusters_once(const cudaLaunchConfig_t& cfg, int cs, int fallback) {
    static std::atomic<int> cache[64][3];  // 0 = not yet queried; cs 1, 2, 4
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) dev = -1;
    const int slot = cs >= 4 ? 2 : cs - 1;
    if (dev >= 0) {
        const int v = cache[dev][slot].load(std::memory_order_relaxed);
        if (v > 0) return v;
    }
    int n = 0;
    if (cudaOccupancyMaxActiveClusters(&n, Kernel, &cfg) != cudaSuccess || n < 1) return fallback;
    if (dev >= 0) cache[dev][slot].store(n, std::memory_order_relaxed);
    return n;
}

}  // namespace tda
