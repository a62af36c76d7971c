// api.cu -- the extern "C" entry points of libtda.so (include/tda.h):
// host-side argument validation, route selection and kernel dispatch.
#include <stdarg.h>
#include <stdio.h>
#include <string.h>

#include <cmath>
#include <atomic>
#include <mutex>

#include "tda_internal.cuh"

namespace tda {

static thread_local char g_msg[512] = "";

tda_status fail(tda_status st, const char* fmt, ...) {
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(g_msg, sizeof(g_msg), fmt, ap);
    va_end(ap);
    return st;
}

tda_status cuda_check(cudaError_t e, const char* what) {
    if (e == cudaSuccess) return TDA_OK;
    return fail(TDA_ERR_CUDA, "%s: %s (%s)", what, cudaGetErrorName(e), cudaGetErrorString(e));
}

static std::atomic<uint64_t> g_launches{0};
void note_launches(uint64_t n) { g_launches.fetch_add(n, std::memory_order_relaxed); }

static std::atomic<int> g_sm_budget{0};
int sm_budget() { return g_sm_budget.load(std::memory_order_relaxed); }

// The device error word: bounded waits that expire OR bits into it.
__device__ unsigned int g_error_word;

unsigned int* device_error_word() {
    static std::mutex mu;
    static unsigned int* cache[64] = {};
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return nullptr;
    std::lock_guard<std::mutex> lock(mu);
    if (!cache[dev]) {
        void* p = nullptr;
        if (cudaGetSymbolAddress(&p, g_error_word) != cudaSuccess) return nullptr;
        cache[dev] = (unsigned int*)p;
    }
    return cache[dev];
}

// ---------------------------------------------------------------------------
// Route cost model (Sec. 3.2, App. A.4, Table 2): flop counts at 2 flops per
// multiply-add, or, after calibration, estimated seconds.
// ---------------------------------------------------------------------------
static std::mutex g_route_mu;
static int g_route_model = 0;
// measured flop/s: [0] factored projection, [1] materialising DW, [2] Gram
// route on bf16 factors (tensor cores), [3] Gram route on fp32 factors
// (projected factors, CUDA cores), [4] projecting a materialised DW with the
// signs, [5] Frobenius inner products of materialised DW
constexpr int kNumRates = 6;
static double g_rate[kNumRates] = {0, 0, 0, 0, 0, 0};
static double g_bw = 0;               // bytes/s

struct RouteCounts {
    double flops[3];
    double bytes[3];
    int gram_rate;   // which measured rate the Gram route runs at (2 or 3)
    double build;    // the materialise route's DW construction flops (the rest of flops[1] runs at post_rate)
    int post_rate;   // 4 (sign projection of DW) or 5 (Frobenius inner products)
};

void set_route_rates(const double* rate, double bw) {
    std::lock_guard<std::mutex> lock(g_route_mu);
    for (int r = 0; r < kNumRates; ++r) g_rate[r] = rate[r];
    g_bw = bw;
    g_route_model = (rate[0] > 0 && bw > 0) ? 1 : 0;
}

static RouteCounts route_counts(const tda_layer_desc& L, tda_op op, int64_t n1, int64_t n2,
                                tda_dtype dt) {
    const double B1 = (double)n1, B2 = (double)n2, T = (double)L.T;
    const double Ni = (double)L.d_in, No = (double)L.d_out, ka = (double)L.k_in, kg = (double)L.k_out;
    const double el = dt == TDA_F32 ? 4.0 : 2.0;
    const double factors = T * (Ni + No) * el;  // one example's factor bytes
    const double proj = 2.0 * T * (Ni * ka + No * kg);
    const double contract = 2.0 * T * ka * kg;
    const double build = 2.0 * T * Ni * No;
    const double dense = 2.0 * No * Ni * ka + 2.0 * No * ka * kg;
    RouteCounts c;
    // the unprojected Gram of bf16 factors runs on tensor cores when T is a power of two
    c.gram_rate = (op == TDA_OP_SIMILARITY_EXACT && dt == TDA_BF16 && L.T > 0 && (L.T & (L.T - 1)) == 0 &&
                   L.d_in % 8 == 0 && L.d_out % 8 == 0)
                      ? 2
                      : 3;
    c.build = (op == TDA_OP_PROJECT || op == TDA_OP_NORM_PROJECTED || op == TDA_OP_NORM_EXACT ? B1 : B1 + B2) * build;
    c.post_rate = (op == TDA_OP_SIMILARITY_EXACT || op == TDA_OP_NORM_EXACT) ? 5 : 4;
    if (op == TDA_OP_PROJECT) {
        c.flops[0] = B1 * (proj + contract);
        c.flops[1] = B1 * (build + dense);
        c.flops[2] = -1;
        c.bytes[0] = B1 * (factors + 4.0 * ka * kg);
        c.bytes[1] = B1 * (factors + 8.0 * Ni * No + 4.0 * ka * kg);
        c.bytes[2] = -1;
    } else if (op == TDA_OP_SIMILARITY_PROJECTED) {
        c.flops[0] = (B1 + B2) * (proj + contract) + B1 * B2 * 2.0 * ka * kg;
        c.flops[1] = (B1 + B2) * (build + dense) + B1 * B2 * 2.0 * ka * kg;
        c.flops[2] = (B1 + B2) * proj + B1 * B2 * 2.0 * T * T * (ka + kg);
        c.bytes[0] = (B1 + B2) * (factors + 4.0 * ka * kg);
        c.bytes[1] = (B1 + B2) * (factors + 8.0 * Ni * No);
        c.bytes[2] = (B1 + B2) * factors + B1 * B2 * 4.0 * T * (ka + kg);
    } else if (op == TDA_OP_SIMILARITY_EXACT) {
        c.flops[0] = -1;
        c.flops[1] = (B1 + B2) * build + B1 * B2 * 2.0 * Ni * No;
        c.flops[2] = B1 * B2 * 2.0 * T * T * (Ni + No);
        c.bytes[0] = -1;
        c.bytes[1] = (B1 + B2) * (factors + 4.0 * Ni * No);
        c.bytes[2] = B1 * B2 * factors;
    } else if (op == TDA_OP_NORM_PROJECTED) {
        c.flops[0] = B1 * (proj + contract + 2.0 * ka * kg);
        c.flops[1] = B1 * (build + dense + 2.0 * ka * kg);
        c.flops[2] = B1 * (proj + 2.0 * T * T * (ka + kg));
        c.bytes[0] = B1 * (factors + 8.0 * ka * kg);
        c.bytes[1] = B1 * (factors + 8.0 * Ni * No);
        c.bytes[2] = B1 * (factors + 8.0 * T * (ka + kg));
    } else {
        c.flops[0] = -1;
        c.flops[1] = B1 * (build + 2.0 * Ni * No);
        c.flops[2] = B1 * 2.0 * T * T * (Ni + No);
        c.bytes[0] = -1;
        c.bytes[1] = B1 * (factors + 8.0 * Ni * No);
        c.bytes[2] = B1 * factors;
    }
    return c;
}

static tda_status validate_layer(const tda_layer_desc* L, bool need_k) {
    if (!L) return fail(TDA_ERR_INVALID_ARG, "layer descriptor is NULL");
    if (L->d_in < 1 || L->d_out < 1 || L->T < 0)
        return fail(TDA_ERR_INVALID_ARG, "bad layer sizes d_in=%lld d_out=%lld T=%lld",
                    (long long)L->d_in, (long long)L->d_out, (long long)L->T);
    if (L->kind != TDA_PROJ_RADEMACHER && L->kind != TDA_PROJ_IDENTITY)
        return fail(TDA_ERR_INVALID_ARG, "bad projection kind %d", L->kind);
    if (need_k) {
        if (L->k_in < 1 || L->k_out < 1)
            return fail(TDA_ERR_INVALID_ARG, "bad projection dims k_in=%d k_out=%d", L->k_in, L->k_out);
        if (L->kind == TDA_PROJ_IDENTITY && (L->k_in != L->d_in || L->k_out != L->d_out))
            return fail(TDA_ERR_INVALID_ARG, "identity projection needs k_in == d_in, k_out == d_out");
    }
    return TDA_OK;
}

static tda_status validate_factors(const tda_layer_desc* L, tda_dtype dt, const void* A,
                                   const void* B, int64_t n, const char* who) {
    if (dt != TDA_F32 && dt != TDA_BF16)
        return fail(TDA_ERR_INVALID_ARG, "%s: dtype must be TDA_F32 or TDA_BF16", who);
    if (n < 0) return fail(TDA_ERR_INVALID_ARG, "%s: negative example count", who);
    if (n > 0 && L->T > 0) {
        if (!A || !B) return fail(TDA_ERR_INVALID_ARG, "%s: NULL factor pointer", who);
        if (((uintptr_t)A & 15) || ((uintptr_t)B & 15))
            return fail(TDA_ERR_INVALID_ARG, "%s: factors must be 16-byte aligned", who);
        const int64_t q = dt == TDA_BF16 ? 8 : 4;
        if (L->d_in % q || L->d_out % q)
            return fail(TDA_ERR_INVALID_ARG, "%s: d_in and d_out must be multiples of %lld", who,
                        (long long)q);
    }
    return TDA_OK;
}

static tda_route_id choose(const RouteCounts& c, double* cost_out) {
    double cost[3];
    std::lock_guard<std::mutex> lock(g_route_mu);
    for (int r = 0; r < 3; ++r) {
        if (c.flops[r] < 0) {
            cost[r] = -1;
        } else if (g_route_model == 1 && r == 1 && g_rate[1] > 0 && g_rate[c.post_rate] > 0 && g_bw > 0) {
            // materialise: DW construction and its use run on different kernels
            cost[r] = std::fmax(c.build / g_rate[1] + (c.flops[1] - c.build) / g_rate[c.post_rate], c.bytes[r] / g_bw);
        } else if (g_route_model == 1 && g_rate[r == 2 ? c.gram_rate : r] > 0 && g_bw > 0) {
            cost[r] = std::fmax(c.flops[r] / g_rate[r == 2 ? c.gram_rate : r], c.bytes[r] / g_bw);
        } else {
            cost[r] = c.flops[r];
        }
    }
    static const int pref[3] = {TDA_ROUTE_GRAM, TDA_ROUTE_FACTORED, TDA_ROUTE_MATERIALIZE};
    int best = -1;
    for (int p = 0; p < 3; ++p) {
        const int r = pref[p];
        if (cost[r] < 0) continue;
        if (best < 0 || cost[r] < cost[best]) best = r;
    }
    if (cost_out)
        for (int r = 0; r < 3; ++r) cost_out[r] = cost[r];
    return (tda_route_id)best;
}

}  // namespace tda

using namespace tda;

extern "C" {

const char* tda_last_error(void) { return g_msg; }

int32_t tda_version(void) { return 100; }

uint64_t tda_launch_count(void) { return g_launches.load(std::memory_order_relaxed); }

tda_status tda_set_sm_budget(int32_t n_sms) {
    g_msg[0] = 0;
    if (n_sms < 0) return fail(TDA_ERR_INVALID_ARG, "tda_set_sm_budget: negative n_sms");
    g_sm_budget.store(n_sms, std::memory_order_relaxed);
    return TDA_OK;
}

int32_t tda_get_sm_budget(void) { return g_sm_budget.load(std::memory_order_relaxed); }

tda_status tda_proj_entries(uint64_t seed, uint32_t layer, int32_t side, int32_t kind, int64_t rows,
                            int32_t cols, int8_t* out, void* stream) {
    g_msg[0] = 0;
    if (side != 0 && side != 1) return fail(TDA_ERR_INVALID_ARG, "side must be 0 or 1");
    if (kind != TDA_PROJ_RADEMACHER && kind != TDA_PROJ_IDENTITY)
        return fail(TDA_ERR_INVALID_ARG, "bad projection kind %d", kind);
    if (rows < 0 || cols < 1 || cols > 1024) return fail(TDA_ERR_INVALID_ARG, "bad rows/cols");
    if (rows > 0 && !out) return fail(TDA_ERR_INVALID_ARG, "out is NULL");
    return cuda_check(launch_proj_entries(side_key(seed, layer, side), kind, rows, cols, out,
                                          (cudaStream_t)stream),
                      "tda_proj_entries launch");
}

tda_status tda_route(const tda_layer_desc* L, tda_op op, int64_t n1, int64_t n2, tda_dtype dtype,
                     tda_route_id* chosen, double* cost_out) {
    g_msg[0] = 0;
    if (op < TDA_OP_PROJECT || op > TDA_OP_NORM_EXACT) return fail(TDA_ERR_INVALID_ARG, "bad op %d", (int)op);
    tda_status st = validate_layer(L, op != TDA_OP_SIMILARITY_EXACT && op != TDA_OP_NORM_EXACT);
    if (st) return st;
    if (n1 < 0 || n2 < 0) return fail(TDA_ERR_INVALID_ARG, "negative batch size");
    if (!chosen) return fail(TDA_ERR_INVALID_ARG, "chosen is NULL");
    *chosen = choose(route_counts(*L, op, n1, n2, dtype), cost_out);
    return TDA_OK;
}

tda_status tda_route_set_model(int32_t model) {
    g_msg[0] = 0;
    if (model != 0 && model != 1) return fail(TDA_ERR_INVALID_ARG, "model must be 0 or 1");
    std::lock_guard<std::mutex> lock(g_route_mu);
    if (model == 1 && !(g_rate[0] > 0 && g_bw > 0))
        return fail(TDA_ERR_INVALID_ARG, "time model needs tda_route_calibrate() first");
    g_route_model = model;
    return TDA_OK;
}

static size_t simproj_ws(const tda_layer_desc& L, int64_t n_q, int64_t chunk, tda_route_id route);
static size_t norms_ws(const tda_layer_desc& L, tda_op op, int64_t chunk, tda_route_id route);

tda_status tda_workspace_size(tda_op op, const tda_layer_desc* L, tda_dtype dtype, int64_t n1,
                              int64_t n2, tda_route_id route, size_t* bytes) {
    g_msg[0] = 0;
    if (!bytes) return fail(TDA_ERR_INVALID_ARG, "bytes is NULL");
    *bytes = 0;
    tda_status st = validate_layer(L, op != TDA_OP_SIMILARITY_EXACT && op != TDA_OP_NORM_EXACT);
    if (st) return st;
    if (route == TDA_ROUTE_AUTO) {
        st = tda_route(L, op, n1, n2, dtype, &route, nullptr);
        if (st) return st;
    }
    if (op == TDA_OP_PROJECT) {
        if (route == TDA_ROUTE_MATERIALIZE) *bytes = materialize_ws_bytes_per_example(*L);
        // optional for the factored route on the tensor cores: balanced token-tile ranges
        // (and for k = 128 precomputed sign tiles)
        if (route == TDA_ROUTE_FACTORED && dtype == TDA_BF16 && L->k_in == L->k_out && L->kind == TDA_PROJ_RADEMACHER &&
            (L->k_in == 16 || L->k_in == 32 || L->k_in == 64 || L->k_in == 128))
            *bytes = project_tc_ws_bytes(*L);
        return TDA_OK;
    }
    if (op == TDA_OP_SIMILARITY_EXACT) {
        if (route == TDA_ROUTE_MATERIALIZE) *bytes = similarity_materialize_ws_bytes(*L, n1, 1);
        return TDA_OK;
    }
    if (op == TDA_OP_SIMILARITY_PROJECTED) {
        *bytes = simproj_ws(*L, n1, 1, route);
        return TDA_OK;
    }
    if (op == TDA_OP_NORM_PROJECTED) {
        *bytes = norms_ws(*L, op, 1, route);
        return TDA_OK;
    }
    if (op == TDA_OP_NORM_EXACT) {
        *bytes = norms_ws(*L, op, 1, route);
        return TDA_OK;
    }
    return fail(TDA_ERR_UNSUPPORTED, "no workspace query for op %d", (int)op);
}

tda_status tda_project(const tda_layer_desc* L, tda_dtype dtype, const void* A, const void* B,
                       int64_t N, float* phi, int64_t ld_phi, tda_route_id route, void* ws,
                       size_t ws_bytes, void* stream) {
    g_msg[0] = 0;
    tda_status st = validate_layer(L, true);
    if (st) return st;
    if ((st = validate_factors(L, dtype, A, B, N, "tda_project"))) return st;
    const int64_t D = (int64_t)L->k_in * L->k_out;
    if (N > 0 && !phi) return fail(TDA_ERR_INVALID_ARG, "phi is NULL");
    if (ld_phi < D) return fail(TDA_ERR_INVALID_ARG, "ld_phi (%lld) < k_in*k_out (%lld)",
                                (long long)ld_phi, (long long)D);
    if (N > 2147483647LL) return fail(TDA_ERR_INVALID_ARG, "N too large");
    if (route == TDA_ROUTE_AUTO) {
        tda_route_id r;
        if ((st = tda_route(L, TDA_OP_PROJECT, N, 0, dtype, &r, nullptr))) return st;
        route = r;
    }
    cudaStream_t s = (cudaStream_t)stream;
    if (N == 0) return TDA_OK;
    if (L->T == 0) return cuda_check(cudaMemset2DAsync(phi, ld_phi * 4, 0, D * 4, N, s), "zero phi");
    if (route == TDA_ROUTE_FACTORED) {
        if (dtype == TDA_BF16 && project_tc_plain_supported(*L, A, B)) {
            unsigned int* err = device_error_word();
            if (!err) return fail(TDA_ERR_CUDA, "cannot resolve the device error word");
            return cuda_check(launch_project_tc(*L, A, B, N, phi, ld_phi, err, s, ws, ws_bytes), "project (tcgen05)");
        }
        return cuda_check(launch_project_simt(*L, dtype, A, B, N, phi, ld_phi, s), "project (simt)");
    }
    if (route == TDA_ROUTE_MATERIALIZE) {
        const size_t need = materialize_ws_bytes_per_example(*L);
        if (!ws || ws_bytes < need)
            return fail(TDA_ERR_WORKSPACE, "materialise route needs >= %zu bytes of ws, got %zu", need,
                        ws_bytes);
        return cuda_check(launch_project_materialized(*L, dtype, A, B, N, phi, ld_phi, ws, ws_bytes, s),
                          "project (materialise)");
    }
    return fail(TDA_ERR_UNSUPPORTED, "route %d cannot produce projected features", (int)route);
}

int32_t tda_project_engine(const tda_layer_desc* L, tda_dtype dtype, const void* A, const void* B) {
    g_msg[0] = 0;
    if (validate_layer(L, true) || validate_factors(L, dtype, A, B, 1, "tda_project_engine")) return -1;
    return (dtype == TDA_BF16 && project_tc_plain_supported(*L, A, B)) ? 1 : 0;
}

tda_status tda_similarity_exact(const tda_layer_desc* L, tda_dtype dtype, const void* Aq,
                                const void* Bq, int64_t n_q, const void* At, const void* Bt,
                                int64_t n_t, float* S, int64_t ld_S, float beta, tda_route_id route,
                                void* ws, size_t ws_bytes, void* stream) {
    g_msg[0] = 0;
    tda_status st = validate_layer(L, false);
    if (st) return st;
    if ((st = validate_factors(L, dtype, Aq, Bq, n_q, "tda_similarity_exact (queries)"))) return st;
    if ((st = validate_factors(L, dtype, At, Bt, n_t, "tda_similarity_exact (train)"))) return st;
    if (n_q > 65535) return fail(TDA_ERR_INVALID_ARG, "n_q must be <= 65535");
    if (n_q > 0 && n_t > 0 && !S) return fail(TDA_ERR_INVALID_ARG, "S is NULL");
    if (ld_S < n_t) return fail(TDA_ERR_INVALID_ARG, "ld_S < n_t");
    if (route == TDA_ROUTE_AUTO) {
        tda_route_id r;
        if ((st = tda_route(L, TDA_OP_SIMILARITY_EXACT, n_q, n_t, dtype, &r, nullptr))) return st;
        route = r;
    }
    cudaStream_t s = (cudaStream_t)stream;
    if (n_q == 0 || n_t == 0) return TDA_OK;
    if (L->T == 0) {
        // DW = 0: the inner products are 0
        return cuda_check(launch_score(S, TDA_F32, n_q, 0, S, n_t, 0, 0, S, ld_S, beta, s), "zero S");
    }
    if (route == TDA_ROUTE_GRAM) {
        if (gram_tc_supported(*L, dtype, Aq, Bq, At, Bt)) {
            unsigned int* err = device_error_word();
            if (!err) return fail(TDA_ERR_CUDA, "device error word unavailable");
            return cuda_check(launch_gram_tc(*L, Aq, Bq, n_q, At, Bt, n_t, S, ld_S, beta, 1.f, err, s),
                              "similarity (gram, tensor cores)");
        }
        return cuda_check(launch_similarity_gram(*L, dtype, Aq, Bq, n_q, At, Bt, n_t, S, ld_S, beta, s),
                          "similarity (gram)");
    }
    if (route == TDA_ROUTE_MATERIALIZE) {
        const size_t need = similarity_materialize_ws_bytes(*L, n_q, 1);
        if (!ws || ws_bytes < need)
            return fail(TDA_ERR_WORKSPACE, "materialise route needs >= %zu bytes of ws, got %zu", need,
                        ws_bytes);
        return cuda_check(launch_similarity_materialized(*L, dtype, Aq, Bq, n_q, At, Bt, n_t, S, ld_S,
                                                         beta, ws, ws_bytes, s),
                          "similarity (materialise)");
    }
    return fail(TDA_ERR_UNSUPPORTED, "route %d cannot produce exact similarities", (int)route);
}

// Workspace of tda_similarity_projected for a train chunk of `chunk` examples.
static size_t simproj_ws(const tda_layer_desc& L, int64_t n_q, int64_t chunk, tda_route_id route) {
    const size_t D = (size_t)L.k_in * (size_t)L.k_out;
    if (route == TDA_ROUTE_GRAM) return project_factors_bytes_per_example(L) * (size_t)(n_q + chunk);
    size_t b = sizeof(float) * D * (size_t)(n_q + chunk);
    if (route == TDA_ROUTE_MATERIALIZE) b += materialize_ws_bytes_per_example(L);
    return b;
}

tda_status tda_similarity_projected(const tda_layer_desc* L, tda_dtype dtype, const void* Aq, const void* Bq,
                                    int64_t n_q, const void* At, const void* Bt, int64_t n_t, float* S,
                                    int64_t ld_S, float beta, tda_route_id route, void* ws, size_t ws_bytes,
                                    void* stream) {
    g_msg[0] = 0;
    tda_status st = validate_layer(L, true);
    if (st) return st;
    if ((st = validate_factors(L, dtype, Aq, Bq, n_q, "tda_similarity_projected (queries)"))) return st;
    if ((st = validate_factors(L, dtype, At, Bt, n_t, "tda_similarity_projected (train)"))) return st;
    if (n_q > 65535) return fail(TDA_ERR_INVALID_ARG, "n_q must be <= 65535");
    if (n_q > 0 && n_t > 0 && !S) return fail(TDA_ERR_INVALID_ARG, "S is NULL");
    if (ld_S < n_t) return fail(TDA_ERR_INVALID_ARG, "ld_S < n_t");
    if (route == TDA_ROUTE_AUTO) {
        tda_route_id r;
        if ((st = tda_route(L, TDA_OP_SIMILARITY_PROJECTED, n_q, n_t, dtype, &r, nullptr))) return st;
        route = r;
    }
    if (route != TDA_ROUTE_FACTORED && route != TDA_ROUTE_MATERIALIZE && route != TDA_ROUTE_GRAM)
        return fail(TDA_ERR_INVALID_ARG, "bad route %d", (int)route);
    cudaStream_t s = (cudaStream_t)stream;
    if (n_q == 0 || n_t == 0) return TDA_OK;
    const size_t need = simproj_ws(*L, n_q, 1, route);
    if (!ws || ws_bytes < need)
        return fail(TDA_ERR_WORKSPACE, "tda_similarity_projected needs >= %zu bytes of ws, got %zu", need, ws_bytes);
    if ((uintptr_t)ws & 255) return fail(TDA_ERR_INVALID_ARG, "ws must be 256-byte aligned");
    const int64_t D = (int64_t)L->k_in * L->k_out;
    const size_t el = dtype == TDA_F32 ? 4 : 2;
    const size_t a_ex = (size_t)L->T * L->d_in * el, b_ex = (size_t)L->T * L->d_out * el;
    if (route == TDA_ROUTE_GRAM) {
        const size_t per = project_factors_bytes_per_example(*L);
        float* Yq = (float*)ws;
        float* Yt = (float*)((char*)ws + per * (size_t)n_q);
        int64_t chunk = (int64_t)((ws_bytes - per * (size_t)n_q) / per);
        if (chunk > n_t) chunk = n_t;
        if (chunk > 65535) chunk = 65535;
        if ((st = cuda_check(launch_project_factors(*L, dtype, Aq, Bq, 0, n_q, Yq, s), "project factors (queries)")))
            return st;
        for (int64_t i0 = 0; i0 < n_t; i0 += chunk) {
            const int64_t c = (n_t - i0) < chunk ? (n_t - i0) : chunk;
            if ((st = cuda_check(launch_project_factors(*L, dtype, At, Bt, i0, c, Yt, s), "project factors (train)")))
                return st;
            if ((st = cuda_check(launch_gram_projected(*L, Yq, n_q, Yt, c, S + i0, ld_S, beta, s), "gram (projected)")))
                return st;
        }
        return TDA_OK;
    }
    // routes a and b: features of the queries, then of train chunks, then scores
    const size_t mat = route == TDA_ROUTE_MATERIALIZE ? materialize_ws_bytes_per_example(*L) : 0;
    float* Fq = (float*)ws;
    float* Ft = Fq + (size_t)n_q * D;
    int64_t chunk = (int64_t)((ws_bytes - mat - sizeof(float) * (size_t)D * (size_t)n_q) / (sizeof(float) * (size_t)D));
    if (chunk > n_t) chunk = n_t;
    void* mws = route == TDA_ROUTE_MATERIALIZE ? (void*)(Ft + (size_t)chunk * D) : nullptr;
    if ((st = tda_project(L, dtype, Aq, Bq, n_q, Fq, D, route, mws, mat, stream))) return st;
    for (int64_t i0 = 0; i0 < n_t; i0 += chunk) {
        const int64_t c = (n_t - i0) < chunk ? (n_t - i0) : chunk;
        if ((st = tda_project(L, dtype, (const char*)At + (size_t)i0 * a_ex, (const char*)Bt + (size_t)i0 * b_ex, c, Ft,
                              D, route, mws, mat, stream)))
            return st;
        if ((st = cuda_check(launch_score(Fq, TDA_F32, n_q, D, Ft, c, D, D, S + i0, ld_S, beta, s), "score")))
            return st;
    }
    return TDA_OK;
}

// Workspace of tda_norms for `chunk` examples at a time.
static size_t norms_ws(const tda_layer_desc& L, tda_op op, int64_t chunk, tda_route_id route) {
    if (op == TDA_OP_NORM_EXACT) {
        if (route == TDA_ROUTE_GRAM) return 0;
        return sizeof(float) * (size_t)(L.d_out * L.d_in) * (size_t)chunk;
    }
    if (route == TDA_ROUTE_GRAM) return project_factors_bytes_per_example(L) * (size_t)chunk;
    size_t b = sizeof(float) * (size_t)L.k_in * (size_t)L.k_out * (size_t)chunk;
    if (route == TDA_ROUTE_MATERIALIZE) b += (materialize_ws_bytes_per_example(L) + 255) & ~(size_t)255;
    return b;
}

tda_status tda_norms(tda_op op, const tda_layer_desc* L, tda_dtype dtype, const void* A, const void* B, int64_t N,
                     float* out, tda_route_id route, void* ws, size_t ws_bytes, void* stream) {
    g_msg[0] = 0;
    if (op != TDA_OP_NORM_PROJECTED && op != TDA_OP_NORM_EXACT)
        return fail(TDA_ERR_INVALID_ARG, "op must be TDA_OP_NORM_PROJECTED or TDA_OP_NORM_EXACT");
    tda_status st = validate_layer(L, op == TDA_OP_NORM_PROJECTED);
    if (st) return st;
    if ((st = validate_factors(L, dtype, A, B, N, "tda_norms"))) return st;
    if (N > 0 && !out) return fail(TDA_ERR_INVALID_ARG, "out is NULL");
    if (route == TDA_ROUTE_AUTO) {
        tda_route_id r;
        if ((st = tda_route(L, op, N, 0, dtype, &r, nullptr))) return st;
        route = r;
    }
    if (op == TDA_OP_NORM_EXACT && route == TDA_ROUTE_FACTORED)
        return fail(TDA_ERR_UNSUPPORTED, "exact norms have no factored-projection route");
    if (route != TDA_ROUTE_FACTORED && route != TDA_ROUTE_MATERIALIZE && route != TDA_ROUTE_GRAM)
        return fail(TDA_ERR_INVALID_ARG, "bad route %d", (int)route);
    cudaStream_t s = (cudaStream_t)stream;
    if (N == 0) return TDA_OK;
    if (L->T == 0) return cuda_check(cudaMemsetAsync(out, 0, sizeof(float) * (size_t)N, s), "zero norms");
    if (op == TDA_OP_NORM_EXACT && route == TDA_ROUTE_GRAM)
        return cuda_check(launch_gram_self(*L, dtype, A, B, N, L->d_in, L->d_out, 1.f, out, s), "norms (gram)");
    const size_t need = norms_ws(*L, op, 1, route);
    if (!ws || ws_bytes < need)
        return fail(TDA_ERR_WORKSPACE, "tda_norms needs >= %zu bytes of ws, got %zu", need, ws_bytes);
    if ((uintptr_t)ws & 255) return fail(TDA_ERR_INVALID_ARG, "ws must be 256-byte aligned");
    const size_t el = dtype == TDA_F32 ? 4 : 2;
    const size_t a_ex = (size_t)L->T * L->d_in * el, b_ex = (size_t)L->T * L->d_out * el;
    if (op == TDA_OP_NORM_EXACT) {  // materialise DW per example, sum of squares
        const int64_t gsz = L->d_out * L->d_in;
        int64_t chunk = (int64_t)(ws_bytes / (sizeof(float) * (size_t)gsz));
        if (chunk > N) chunk = N;
        if (chunk > 65535) chunk = 65535;
        for (int64_t i0 = 0; i0 < N; i0 += chunk) {
            const int64_t c = (N - i0) < chunk ? (N - i0) : chunk;
            if ((st = cuda_check(launch_materialize_G(*L, dtype, A, B, i0, c, (float*)ws, s), "materialise")))
                return st;
            if ((st = cuda_check(launch_row_sq_norms((const float*)ws, c, gsz, gsz, out + i0, s), "norms")))
                return st;
        }
        return TDA_OK;
    }
    if (route == TDA_ROUTE_GRAM) {  // Eq. 4 on the projected factors of each example with itself
        const size_t per = project_factors_bytes_per_example(*L);
        int64_t chunk = (int64_t)(ws_bytes / per);
        if (chunk > N) chunk = N;
        if (chunk > 65535) chunk = 65535;
        const float sc = projection_scale(*L);
        for (int64_t i0 = 0; i0 < N; i0 += chunk) {
            const int64_t c = (N - i0) < chunk ? (N - i0) : chunk;
            float* Y = (float*)ws;
            if ((st = cuda_check(launch_project_factors(*L, dtype, A, B, i0, c, Y, s), "project factors"))) return st;
            if ((st = cuda_check(launch_gram_self(*L, TDA_F32, Y, Y + c * L->T * L->k_in, c, L->k_in, L->k_out,
                                                  sc * sc, out + i0, s),
                                 "norms (projected gram)")))
                return st;
        }
        return TDA_OK;
    }
    // routes a and b: features in ws, then row sums of squares
    const int64_t D = (int64_t)L->k_in * L->k_out;
    // [materialisation scratch, 256-aligned | features of `chunk` examples]
    const size_t mat =
        route == TDA_ROUTE_MATERIALIZE ? (materialize_ws_bytes_per_example(*L) + 255) & ~(size_t)255 : 0;
    int64_t chunk = (int64_t)((ws_bytes - mat) / (sizeof(float) * (size_t)D));
    if (chunk > N) chunk = N;
    void* mws = mat ? ws : nullptr;
    float* F = (float*)((char*)ws + mat);
    for (int64_t i0 = 0; i0 < N; i0 += chunk) {
        const int64_t c = (N - i0) < chunk ? (N - i0) : chunk;
        if ((st = tda_project(L, dtype, (const char*)A + (size_t)i0 * a_ex, (const char*)B + (size_t)i0 * b_ex, c, F, D,
                              route, mws, mat, stream)))
            return st;
        if ((st = cuda_check(launch_row_sq_norms(F, c, D, D, out + i0, s), "norms"))) return st;
    }
    return TDA_OK;
}

tda_status tda_cosine(float* S, int64_t n_q, int64_t n_t, int64_t ld_S, const float* nq, const float* nt,
                      void* stream) {
    g_msg[0] = 0;
    if (n_q < 0 || n_t < 0 || ld_S < n_t) return fail(TDA_ERR_INVALID_ARG, "bad sizes");
    if (n_q > 0 && n_t > 0 && (!S || !nq || !nt)) return fail(TDA_ERR_INVALID_ARG, "NULL argument");
    return cuda_check(launch_cosine(S, n_q, n_t, ld_S, nq, nt, (cudaStream_t)stream), "cosine");
}

// ---------------------------------------------------------------- token scores / masks
size_t tda_token_scores_workspace_size(const tda_layer_desc* L) {
    if (!L || L->k_in < 1 || L->k_out < 1 || L->T < 0) return 0;
    return (project_factors_bytes_per_example(*L) + 255) & ~(size_t)255;
}

tda_status tda_token_scores(const tda_layer_desc* L, tda_dtype dtype, const void* A, const void* B, int64_t N,
                            const float* R, int64_t n_q, int64_t ld_R, float* out, int64_t ld_q_out, float beta,
                            void* ws, size_t ws_bytes, void* stream) {
    g_msg[0] = 0;
    tda_status st = validate_layer(L, true);
    if (st) return st;
    if ((st = validate_factors(L, dtype, A, B, N, "tda_token_scores"))) return st;
    if (L->k_in > 128 || L->k_out > 128) return fail(TDA_ERR_UNSUPPORTED, "token scores need k_in, k_out <= 128");
    const int64_t D = (int64_t)L->k_in * L->k_out;
    if (n_q < 0) return fail(TDA_ERR_INVALID_ARG, "negative n_q");
    if (N > 0 && n_q > 0 && L->T > 0) {
        if (!R || ld_R < D) return fail(TDA_ERR_INVALID_ARG, "R is NULL or ld_R < k_in*k_out");
        if (!out || ld_q_out < N * L->T) return fail(TDA_ERR_INVALID_ARG, "out is NULL or ld_q_out < N*T");
    }
    const size_t per = project_factors_bytes_per_example(*L);
    if (N == 0 || n_q == 0 || L->T == 0) return TDA_OK;
    if (!ws || ws_bytes < per)
        return fail(TDA_ERR_WORKSPACE, "tda_token_scores needs >= %zu bytes of ws, got %zu", per, ws_bytes);
    cudaStream_t s = (cudaStream_t)stream;
    // The tensor-core contraction (k_in = 32) keeps R's hi and lo halves at the
    // front of the workspace when it has room for them and one example.
    const size_t rsplit = token_tc_split_bytes(L->k_in, L->k_out, n_q);
    const bool tc = token_tc_supported(L->k_in, L->k_out, n_q) && ((uintptr_t)ws & 255) == 0 && ws_bytes >= rsplit + per &&
                    ((uintptr_t)R & 3) == 0;
    const size_t off = tc ? rsplit : 0;
    int64_t chunk = (int64_t)((ws_bytes - off) / per);
    if (chunk > N) chunk = N;
    if (chunk > 65535) chunk = 65535;
    const float scale = projection_scale(*L);
    float* Y = (float*)((char*)ws + off);
    for (int64_t e0 = 0; e0 < N; e0 += chunk) {
        const int64_t c = N - e0 < chunk ? N - e0 : chunk;
        if ((st = cuda_check(launch_project_factors(*L, dtype, A, B, e0, c, Y, s), "project factors"))) return st;
        const float* Yb = Y + c * L->T * L->k_in;
        if (tc)
            st = cuda_check(launch_token_scores_tc(Y, Yb, c, L->T, L->k_in, L->k_out, R, n_q, ld_R, scale, out,
                                                   ld_q_out, e0, beta, (float*)ws, s),
                            "token scores (tensor cores)");
        else
            st = cuda_check(launch_token_scores(Y, Yb, c, L->T, L->k_in, L->k_out, R, n_q, ld_R, scale, out, ld_q_out,
                                                e0, beta, s),
                            "token scores");
        if (st) return st;
    }
    return TDA_OK;
}

tda_status tda_mask_gather(const tda_layer_desc* L, tda_dtype dtype, const void* A, const void* B, int64_t N,
                           const int32_t* rows, const int32_t* cols, int64_t n_coords, float* out, int64_t ld_out,
                           void* stream) {
    g_msg[0] = 0;
    tda_status st = validate_layer(L, false);
    if (st) return st;
    if ((st = validate_factors(L, dtype, A, B, N, "tda_mask_gather"))) return st;
    if (n_coords < 0) return fail(TDA_ERR_INVALID_ARG, "negative n_coords");
    if (N > 0 && n_coords > 0 && (!rows || !cols || !out || ld_out < n_coords))
        return fail(TDA_ERR_INVALID_ARG, "rows/cols/out NULL or ld_out < n_coords");
    if (L->d_in > 65536 || L->d_out > 65536) return fail(TDA_ERR_UNSUPPORTED, "mask gather needs d <= 65536");
    const size_t el = dtype == TDA_F32 ? 4 : 2;
    if (mask_gather_tokens_per_pass(L->d_in, L->d_out, el) < 1)
        return fail(TDA_ERR_UNSUPPORTED, "mask gather needs (d_in + d_out) * sizeof(dtype) <= 48 KiB");
    if (N == 0 || n_coords == 0) return TDA_OK;
    cudaStream_t s = (cudaStream_t)stream;
    if (L->T == 0) {
        for (int64_t n = 0; n < N; ++n)
            if ((st = cuda_check(cudaMemsetAsync(out + n * ld_out, 0, sizeof(float) * (size_t)n_coords, s), "zero")))
                return st;
        return TDA_OK;
    }
    const size_t a_ex = (size_t)L->T * L->d_in * el, b_ex = (size_t)L->T * L->d_out * el;
    for (int64_t e0 = 0; e0 < N; e0 += 65535) {
        const int64_t c = N - e0 < 65535 ? N - e0 : 65535;
        if ((st = cuda_check(launch_mask_gather(*L, dtype, (const char*)A + e0 * a_ex, (const char*)B + e0 * b_ex, c,
                                                rows, cols, n_coords, out + e0 * ld_out, ld_out, s),
                             "mask gather")))
            return st;
    }
    return TDA_OK;
}

// ---------------------------------------------------------------- K-FAC / EK-FAC
static bool kfac_dims_ok(int64_t ka, int64_t kg) { return ka >= 1 && kg >= 1 && ka <= 128 && kg <= 128; }

size_t tda_kfac_state_bytes(int32_t k_in, int32_t k_out) {
    if (!kfac_dims_ok(k_in, k_out)) return 0;
    return kfac_state_bytes(k_in, k_out);
}

// scratch of the K-FAC calls: per-block partial sums (fixed-order reduction)
// and, for tda_kfac_accumulate_factors, one example's projected factors
static size_t kfac_partials_bytes(int64_t ka, int64_t kg) {
    const int64_t kmax2 = (ka > kg ? ka : kg) * (ka > kg ? ka : kg);
    size_t b = sizeof(float) * 304 * (size_t)kmax2;                                      // covariance / EK-FAC partials
    const size_t fused = sizeof(float) * (size_t)project_tc_max_grid() * 2 * (size_t)kmax2;  // fused projection
    if (fused > b) b = fused;
    return (b + 255) & ~(size_t)255;
}

size_t tda_kfac_workspace_size(const tda_layer_desc* L, tda_dtype dtype) {
    (void)dtype;
    if (!L || !kfac_dims_ok(L->k_in, L->k_out) || L->T < 0) return 0;
    return kfac_partials_bytes(L->k_in, L->k_out) + project_factors_bytes_per_example(*L);
}

static tda_status kfac_state_ok(int64_t ka, int64_t kg, const void* state) {
    if (!kfac_dims_ok(ka, kg)) return fail(TDA_ERR_INVALID_ARG, "K-FAC needs 1 <= k_in, k_out <= 128");
    if (!state || ((uintptr_t)state & 15)) return fail(TDA_ERR_INVALID_ARG, "state must be a 16-byte aligned pointer");
    return TDA_OK;
}

tda_status tda_kfac_reset(int32_t n_layers, int32_t k_in, int32_t k_out, void* state, void* stream) {
    g_msg[0] = 0;
    tda_status st = kfac_state_ok(k_in, k_out, state);
    if (st) return st;
    if (n_layers < 1 || n_layers > 65535) return fail(TDA_ERR_INVALID_ARG, "n_layers must be in [1, 65535]");
    return cuda_check(cudaMemsetAsync(state, 0, (size_t)n_layers * kfac_state_bytes(k_in, k_out), (cudaStream_t)stream),
                      "kfac reset");
}

tda_status tda_kfac_accumulate_factors(const tda_layer_desc* L, tda_dtype dtype, const void* A, const void* B,
                                       int64_t N, void* state, void* ws, size_t ws_bytes, void* stream) {
    g_msg[0] = 0;
    tda_status st = validate_layer(L, true);
    if (st) return st;
    if ((st = validate_factors(L, dtype, A, B, N, "tda_kfac_accumulate_factors"))) return st;
    if (L->kind != TDA_PROJ_RADEMACHER && L->kind != TDA_PROJ_IDENTITY) return fail(TDA_ERR_INVALID_ARG, "bad kind");
    if ((st = kfac_state_ok(L->k_in, L->k_out, state))) return st;
    const size_t need = tda_kfac_workspace_size(L, dtype);
    if (!ws || ws_bytes < need)
        return fail(TDA_ERR_WORKSPACE, "tda_kfac_accumulate_factors needs >= %zu bytes of ws, got %zu", need,
                    ws_bytes);
    if ((uintptr_t)ws & 255) return fail(TDA_ERR_INVALID_ARG, "ws must be 256-byte aligned");
    cudaStream_t s = (cudaStream_t)stream;
    double* sd = (double*)state;
    const int64_t ka = L->k_in, kg = L->k_out;
    double* Sa = sd + kfac_offset_sa(ka, kg);
    double* Sg = sd + kfac_offset_sg(ka, kg);
    // Rademacher factors come out of the projection with +-1 signs: 1/k restores P = S / sqrt(k)
    const double sca = L->kind == TDA_PROJ_RADEMACHER ? 1.0 / (double)ka : 1.0;
    const double scg = L->kind == TDA_PROJ_RADEMACHER ? 1.0 / (double)kg : 1.0;
    const size_t pbytes = kfac_partials_bytes(ka, kg);
    float* part = (float*)ws;
    float* Y = (float*)((char*)ws + pbytes);
    if (N == 0 || L->T == 0)
        return cuda_check(launch_kfac_cov(Y, 0, (int)ka, Sa, sca, sd, (double)N * (double)L->T, part, s),
                          "kfac token count");
    const size_t per = project_factors_bytes_per_example(*L);
    int64_t chunk = (int64_t)((ws_bytes - pbytes) / per);
    if (chunk > N) chunk = N;
    if (chunk > 65535) chunk = 65535;
    for (int64_t e0 = 0; e0 < N; e0 += chunk) {
        const int64_t c = N - e0 < chunk ? N - e0 : chunk;
        if ((st = cuda_check(launch_project_factors(*L, dtype, A, B, e0, c, Y, s), "project factors"))) return st;
        const int64_t rows = c * L->T;
        if ((st = cuda_check(launch_kfac_cov(Y, rows, (int)ka, Sa, sca, sd, (double)rows, part, s), "cov a")))
            return st;
        if ((st = cuda_check(launch_kfac_cov(Y + rows * ka, rows, (int)kg, Sg, scg, nullptr, 0.0, part, s),
                             "cov g")))
            return st;
    }
    return TDA_OK;
}

tda_status tda_project_kfac(const tda_layer_desc* L, tda_dtype dtype, const void* A, const void* B, int64_t N,
                            float* phi, int64_t ld_phi, void* state, void* ws, size_t ws_bytes, void* stream) {
    g_msg[0] = 0;
    tda_status st = validate_layer(L, true);
    if (st) return st;
    if ((st = validate_factors(L, dtype, A, B, N, "tda_project_kfac"))) return st;
    if ((st = kfac_state_ok(L->k_in, L->k_out, state))) return st;
    const int64_t D = (int64_t)L->k_in * L->k_out;
    if (N > 0 && (!phi || ld_phi < D)) return fail(TDA_ERR_INVALID_ARG, "phi is NULL or ld_phi < k_in*k_out");
    if (dtype != TDA_BF16 || N == 0 || L->T == 0 || !project_tc_supported(*L, A, B))
        return fail(TDA_ERR_UNSUPPORTED, "tda_project_kfac runs the bf16 tensor-core projection only");
    const size_t need = kfac_partials_bytes(L->k_in, L->k_out);
    if (!ws || ws_bytes < need)
        return fail(TDA_ERR_WORKSPACE, "tda_project_kfac needs >= %zu bytes of ws, got %zu", need, ws_bytes);
    if ((uintptr_t)ws & 255) return fail(TDA_ERR_INVALID_ARG, "ws must be 256-byte aligned");
    unsigned int* err = device_error_word();
    if (!err) return fail(TDA_ERR_CUDA, "device error word unavailable");
    cudaStream_t s = (cudaStream_t)stream;
    float* part = (float*)ws;
    int grid = 0;
    if ((st = cuda_check(launch_project_tc_kfac(*L, A, B, N, phi, ld_phi, part, &grid, err, s), "project+kfac")))
        return st;
    const int64_t k = L->k_in, kk = k * k;
    double* sd = (double*)state;
    const double sc = 1.0 / (double)k;
    if ((st = cuda_check(launch_kfac_sum_partials(part, grid, 2 * kk, kk, sd + kfac_offset_sa(k, k), sc, sd, 0,
                                                  (double)N * (double)L->T, s),
                         "kfac sums a")))
        return st;
    return cuda_check(launch_kfac_sum_partials(part + kk, grid, 2 * kk, kk, sd + kfac_offset_sg(k, k), sc, nullptr, 0,
                                               0.0, s),
                      "kfac sums g");
}

tda_status tda_kfac_eigen(int32_t n_layers, int32_t k_in, int32_t k_out, void* state, void* stream) {
    g_msg[0] = 0;
    tda_status st = kfac_state_ok(k_in, k_out, state);
    if (st) return st;
    if (n_layers < 1 || n_layers > 65535) return fail(TDA_ERR_INVALID_ARG, "n_layers must be in [1, 65535]");
    return cuda_check(launch_kfac_eigen(n_layers, (double*)state, k_in, k_out, (cudaStream_t)stream), "kfac eigen");
}

tda_status tda_kfac_accumulate_eigenvalues(int32_t n_layers, int32_t k_in, int32_t k_out, void* state,
                                           const float* phi, int64_t n, int64_t ld_phi, void* ws, size_t ws_bytes,
                                           void* stream) {
    g_msg[0] = 0;
    tda_status st = kfac_state_ok(k_in, k_out, state);
    if (st) return st;
    if (n_layers < 1 || n_layers > 65535) return fail(TDA_ERR_INVALID_ARG, "n_layers must be in [1, 65535]");
    const int64_t D = (int64_t)k_in * k_out;
    if (n < 0 || (n > 0 && (!phi || ld_phi < (int64_t)n_layers * D)))
        return fail(TDA_ERR_INVALID_ARG, "phi is NULL or ld_phi < n_layers*k_in*k_out");
    const size_t need = kfac_partials_bytes(k_in, k_out);
    if (!ws || ws_bytes < need)
        return fail(TDA_ERR_WORKSPACE, "tda_kfac_accumulate_eigenvalues needs >= %zu bytes of ws, got %zu", need,
                    ws_bytes);
    // every (layer, block) pair writes one partial of D floats into ws
    const int64_t slabs = (int64_t)(ws_bytes / (sizeof(float) * (size_t)D));
    const size_t lbytes = kfac_state_bytes(k_in, k_out);
    for (int32_t l0 = 0; l0 < n_layers;) {
        int32_t nl = n_layers - l0;
        if (nl > slabs) nl = (int32_t)slabs;
        int64_t nblk = slabs / nl;
        if (nblk > 304 / nl) nblk = 304 / nl;
        if (nblk > n) nblk = n;
        if (nblk < 1) nblk = 1;
        if ((st = cuda_check(launch_kfac_ekfac_accum(nl, (double*)((char*)state + (size_t)l0 * lbytes), k_in, k_out,
                                                     phi + (int64_t)l0 * D, n, ld_phi, (float*)ws, (int)nblk,
                                                     (cudaStream_t)stream),
                             "ekfac eigenvalues")))
            return st;
        l0 += nl;
    }
    return TDA_OK;
}

tda_status tda_kfac_apply(int32_t kind, int32_t n_layers, int32_t k_in, int32_t k_out, const void* state,
                          double lambda_abs, double lambda_rel, const float* q, int64_t n_q, int64_t ld_q, float* qhat,
                          int64_t ld_qhat, void* stream) {
    g_msg[0] = 0;
    tda_status st = kfac_state_ok(k_in, k_out, state);
    if (st) return st;
    if (kind != TDA_KFAC && kind != TDA_EKFAC) return fail(TDA_ERR_INVALID_ARG, "kind must be TDA_KFAC or TDA_EKFAC");
    if (n_layers < 1 || n_layers > 65535) return fail(TDA_ERR_INVALID_ARG, "n_layers must be in [1, 65535]");
    const int64_t D = (int64_t)k_in * k_out;
    if (n_q < 0 || n_q > 2147483647LL) return fail(TDA_ERR_INVALID_ARG, "bad n_q");
    if (n_q > 0 && (!q || !qhat || ld_q < n_layers * D || ld_qhat < n_layers * D))
        return fail(TDA_ERR_INVALID_ARG, "q/qhat NULL or leading dimension < n_layers*k_in*k_out");
    return cuda_check(launch_kfac_apply(kind, n_layers, (const double*)state, k_in, k_out, lambda_abs, lambda_rel, q,
                                        n_q, ld_q, qhat, ld_qhat, (cudaStream_t)stream),
                      "kfac apply");
}

size_t tda_precondition_state_bytes(int64_t D, tda_dtype state_dtype) {
    if (D < 1 || (state_dtype != TDA_F32 && state_dtype != TDA_F64)) return 0;
    const size_t el = state_dtype == TDA_F64 ? 8 : 4;
    const size_t nblk = (size_t)((D + 31) / 32);
    const size_t raw = kPcHeaderDoubles * sizeof(double) + ((size_t)D * (size_t)D + nblk * 1024) * el;
    return (raw + 255) & ~(size_t)255;
}

tda_status tda_precondition(int32_t op, int32_t n_layers, int64_t D, tda_dtype state_dtype, void* state,
                            const float* phi, int64_t n, int64_t ld_phi, int64_t n_total,
                            double lambda_abs, double lambda_rel_mean_eig, const float* q,
                            int64_t n_q, int64_t ld_q, void* qhat, int64_t ld_qhat, void* stream) {
    g_msg[0] = 0;
    if (n_layers < 1 || n_layers > 65535) return fail(TDA_ERR_INVALID_ARG, "n_layers must be in [1, 65535]");
    if (D < 1 || D > (1LL << 20)) return fail(TDA_ERR_INVALID_ARG, "D must be in [1, 2^20]");
    if (state_dtype != TDA_F32 && state_dtype != TDA_F64)
        return fail(TDA_ERR_INVALID_ARG, "state dtype must be TDA_F32 or TDA_F64");
    if (!state) return fail(TDA_ERR_INVALID_ARG, "state is NULL");
    if ((uintptr_t)state & 15) return fail(TDA_ERR_INVALID_ARG, "state must be 16-byte aligned");
    const int64_t width = (int64_t)n_layers * D;  // features per row across the layers
    cudaStream_t s = (cudaStream_t)stream;
    switch (op) {
        case TDA_PC_RESET:
            return cuda_check(cudaMemsetAsync(state, 0, (size_t)n_layers * tda_precondition_state_bytes(D, state_dtype), s),
                              "reset state");
        case TDA_PC_FIT_ACCUM:
            if (n < 0) return fail(TDA_ERR_INVALID_ARG, "negative n");
            if (n > 0 && !phi) return fail(TDA_ERR_INVALID_ARG, "phi is NULL");
            if (ld_phi < width) return fail(TDA_ERR_INVALID_ARG, "ld_phi < n_layers*D");
            return cuda_check(launch_pc_fit(n_layers, D, state_dtype, state, phi, n, ld_phi, s), "fit");
        case TDA_PC_FACTOR:
            if (n_total < 1) return fail(TDA_ERR_INVALID_ARG, "n_total must be >= 1");
            if (!(lambda_abs >= 0) || !(lambda_rel_mean_eig >= 0) ||
                !(lambda_abs > 0 || lambda_rel_mean_eig > 0))
                return fail(TDA_ERR_INVALID_ARG, "damping must be >= 0 and not both zero");
            return cuda_check(launch_pc_factor(n_layers, D, state_dtype, state, n_total, lambda_abs,
                                               lambda_rel_mean_eig, s),
                              "factor");
        case TDA_PC_FACTOR_APPLY: {
            if (n_total < 1) return fail(TDA_ERR_INVALID_ARG, "n_total must be >= 1");
            if (!(lambda_abs >= 0) || !(lambda_rel_mean_eig >= 0) ||
                !(lambda_abs > 0 || lambda_rel_mean_eig > 0))
                return fail(TDA_ERR_INVALID_ARG, "damping must be >= 0 and not both zero");
            if (n_q < 0) return fail(TDA_ERR_INVALID_ARG, "negative n_q");
            if (n_q > 0 && (!q || !qhat)) return fail(TDA_ERR_INVALID_ARG, "q/qhat is NULL");
            if (ld_q < width || ld_qhat < width) return fail(TDA_ERR_INVALID_ARG, "ld_q/ld_qhat < n_layers*D");
            if (D > precondition_apply_max_d(state_dtype))
                return fail(TDA_ERR_UNSUPPORTED, "APPLY keeps a query row in shared memory: D > %lld",
                            (long long)precondition_apply_max_d(state_dtype));
            if (n_q == 0)
                return cuda_check(launch_pc_factor(n_layers, D, state_dtype, state, n_total, lambda_abs,
                                                   lambda_rel_mean_eig, s),
                                  "factor");
            return cuda_check(launch_pc_factor_apply(n_layers, D, state_dtype, state, n_total, lambda_abs,
                                                     lambda_rel_mean_eig, q, n_q, ld_q, qhat, ld_qhat, s),
                              "factor + apply");
        }
        case TDA_PC_APPLY: {
            if (n_q < 0) return fail(TDA_ERR_INVALID_ARG, "negative n_q");
            if (n_q > 0 && (!q || !qhat)) return fail(TDA_ERR_INVALID_ARG, "q/qhat is NULL");
            if (ld_q < width || ld_qhat < width) return fail(TDA_ERR_INVALID_ARG, "ld_q/ld_qhat < n_layers*D");
            if (D > precondition_apply_max_d(state_dtype))
                return fail(TDA_ERR_UNSUPPORTED, "APPLY keeps a query row in shared memory: D > %lld",
                            (long long)precondition_apply_max_d(state_dtype));
            return cuda_check(launch_pc_apply(n_layers, D, state_dtype, state, q, n_q, ld_q, qhat, ld_qhat, s),
                              "apply");
        }
        default:
            return fail(TDA_ERR_INVALID_ARG, "bad precondition op %d", op);
    }
}

tda_status tda_precondition_info(int32_t n_layers, int64_t D, tda_dtype state_dtype, const void* state,
                                 double* info, void* stream) {
    g_msg[0] = 0;
    if (!state || !info) return fail(TDA_ERR_INVALID_ARG, "NULL argument");
    if (n_layers < 1) return fail(TDA_ERR_INVALID_ARG, "n_layers must be >= 1");
    const size_t per = tda_precondition_state_bytes(D, state_dtype);
    if (!per) return fail(TDA_ERR_INVALID_ARG, "bad D or state dtype");
    cudaStream_t s = (cudaStream_t)stream;
    double fail_at = 0;
    int fail_layer = -1;
    for (int32_t l = 0; l < n_layers; ++l) {
        double h[kPcHeaderDoubles];
        tda_status st = cuda_check(
            cudaMemcpyAsync(h, (const char*)state + (size_t)l * per, sizeof(h), cudaMemcpyDeviceToHost, s),
            "read header");
        if (st) return st;
        if ((st = cuda_check(cudaStreamSynchronize(s), "sync"))) return st;
        info[4 * l + 0] = h[kPcLambda];
        info[4 * l + 1] = h[kPcMeanEig];
        info[4 * l + 2] = h[kPcFailedPivot];
        info[4 * l + 3] = h[kPcNTotal];
        if (h[kPcFailedPivot] != 0.0 && fail_layer < 0) {
            fail_layer = l;
            fail_at = h[kPcFailedPivot];
        }
    }
    if (fail_layer >= 0)
        return fail(TDA_ERR_NOT_SPD, "layer %d: F + lambda I not positive definite at pivot %.0f", fail_layer,
                    fail_at);
    return TDA_OK;
}

tda_status tda_score(const void* Qhat, tda_dtype q_dtype, int64_t n_q, int64_t ld_q, const float* Phi,
                     int64_t n_t, int64_t ld_phi, int64_t D, float* S, int64_t ld_S, float beta,
                     void* stream) {
    g_msg[0] = 0;
    if (q_dtype != TDA_F32 && q_dtype != TDA_F64)
        return fail(TDA_ERR_INVALID_ARG, "Qhat dtype must be TDA_F32 or TDA_F64");
    if (n_q < 0 || n_t < 0 || D < 0) return fail(TDA_ERR_INVALID_ARG, "negative size");
    if (n_q > 65535LL * 32) return fail(TDA_ERR_INVALID_ARG, "n_q too large");
    if (n_q > 0 && n_t > 0) {
        if (!S) return fail(TDA_ERR_INVALID_ARG, "S is NULL");
        if (D > 0 && (!Qhat || !Phi)) return fail(TDA_ERR_INVALID_ARG, "Qhat/Phi is NULL");
    }
    if (ld_q < D || ld_phi < D || ld_S < n_t) return fail(TDA_ERR_INVALID_ARG, "leading dimension too small");
    if (n_q > 0 && n_t > 0 && score_tc_supported(q_dtype, Qhat, n_q, ld_q, Phi, n_t, ld_phi, D)) {
        unsigned int* err = device_error_word();
        if (!err) return fail(TDA_ERR_CUDA, "cannot resolve the device error word");
        return cuda_check(launch_score_tc((const float*)Qhat, n_q, ld_q, Phi, n_t, ld_phi, D, S, ld_S, beta, err,
                                          (cudaStream_t)stream),
                          "score (tcgen05)");
    }
    return cuda_check(launch_score(Qhat, q_dtype, n_q, ld_q, Phi, n_t, ld_phi, D, S, ld_S, beta,
                                   (cudaStream_t)stream),
                      "score");
}

int32_t tda_similarity_gram_engine(const tda_layer_desc* L, tda_dtype dtype, const void* Aq, const void* Bq,
                                   const void* At, const void* Bt) {
    if (!L || L->T < 1) return 0;
    return gram_tc_supported(*L, dtype, Aq, Bq, At, Bt) ? 1 : 0;
}

int32_t tda_score_engine(const void* Qhat, tda_dtype q_dtype, int64_t n_q, int64_t ld_q, const float* Phi,
                         int64_t n_t, int64_t ld_phi, int64_t D) {
    return score_tc_supported(q_dtype, Qhat, n_q, ld_q, Phi, n_t, ld_phi, D) ? 1 : 0;
}

tda_status tda_topk(const float* S, int64_t n_q, int64_t n_t, int64_t ld_S, int32_t k, int32_t* idx,
                    float* val, void* stream) {
    g_msg[0] = 0;
    if (n_q < 0 || n_t < 0) return fail(TDA_ERR_INVALID_ARG, "negative size");
    if (k < 1 || k > 1024 || k > n_t) return fail(TDA_ERR_INVALID_ARG, "need 1 <= k <= min(n_t, 1024)");
    if (n_t > 0xFFFFFFFFLL) return fail(TDA_ERR_INVALID_ARG, "n_t too large");
    if (ld_S < n_t) return fail(TDA_ERR_INVALID_ARG, "ld_S < n_t");
    if (n_q > 0 && (!S || !idx)) return fail(TDA_ERR_INVALID_ARG, "S/idx is NULL");
    return cuda_check(launch_topk(S, n_q, n_t, ld_S, k, idx, val, (cudaStream_t)stream), "topk");
}

tda_status tda_device_status(void* stream) {
    g_msg[0] = 0;
    tda_status st = cuda_check(cudaStreamSynchronize((cudaStream_t)stream), "stream sync");
    if (st) return st;
    unsigned int w = 0;
    if ((st = cuda_check(cudaMemcpyFromSymbol(&w, g_error_word, sizeof(w)), "read error word"))) return st;
    if (w) {
        unsigned int z = 0;
        cudaMemcpyToSymbol(g_error_word, &z, sizeof(z));
        if (w & kErrTimeout) return fail(TDA_ERR_TIMEOUT, "a device-side bounded wait expired (word %#x)", w);
        return fail(TDA_ERR_CUDA, "device reported an inconsistent launch (word %#x)", w);
    }
    return TDA_OK;
}

}  // extern "C"
