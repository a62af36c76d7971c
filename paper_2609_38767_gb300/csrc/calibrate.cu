// calibrate.cu -- device calibration of the route cost model (Sec. 3.2 and
// App. A.4 estimate costs per layer and op; on a given GPU the routes run at
// different rates, so the estimate becomes seconds = max(flops / rate_route,
// bytes / bandwidth) with rates measured here by short launches of the route
// kernels themselves).
#include <cmath>

#include "tda_internal.cuh"

namespace tda {
void set_route_rates(const double* rate, double bw);
}

using namespace tda;

namespace {

struct EventTimer {
    cudaEvent_t a = nullptr, b = nullptr;
    EventTimer() {
        cudaEventCreate(&a);
        cudaEventCreate(&b);
    }
    ~EventTimer() {
        cudaEventDestroy(a);
        cudaEventDestroy(b);
    }
};

}  // namespace

extern "C" tda_status tda_route_calibrate(void* ws, size_t ws_bytes, void* stream, double* rates_out) {
    if (!ws || ws_bytes < TDA_CALIBRATE_WS_BYTES)
        return fail(TDA_ERR_WORKSPACE, "tda_route_calibrate needs >= %zu bytes of ws",
                    (size_t)TDA_CALIBRATE_WS_BYTES);
    if ((uintptr_t)ws & 255) return fail(TDA_ERR_INVALID_ARG, "ws must be 256-byte aligned");
    cudaStream_t s = (cudaStream_t)stream;
    char* base = (char*)ws;
    tda_status st = cuda_check(cudaMemsetAsync(ws, 0, TDA_CALIBRATE_WS_BYTES, s), "clear ws");
    if (st) return st;

    tda_layer_desc L{};
    L.d_in = 1024;
    L.d_out = 1024;
    L.T = 128;
    L.k_in = 32;
    L.k_out = 32;
    L.seed = 0;
    L.layer = 0;
    L.kind = TDA_PROJ_RADEMACHER;
    const int64_t Nf = 512;  // factored: 2 x 128 MiB of bf16 factors
    const size_t fbytes = (size_t)Nf * L.T * L.d_in * 2;
    void* A = base;
    void* B = base + fbytes;
    float* phi = (float*)(base + 2 * fbytes);
    char* rest = base + 2 * fbytes + (size_t)Nf * 1024 * 4;
    const size_t rest_bytes = TDA_CALIBRATE_WS_BYTES - (size_t)(rest - base) - (1u << 20);
    float* S = (float*)(base + TDA_CALIBRATE_WS_BYTES - (1u << 20));

    EventTimer ev;
    // kinds: 0 factored projection, 1 DW construction, 2 Gram (bf16), 3 Gram (projected factors),
    // 4 materialise route of the projection (construction + sign projection), 5 Frobenius dots
    constexpr int kKinds = 6;
    double secs[kKinds] = {0, 0, 0, 0, 0, 0};
    const double T = 128, d = 1024, k = 32;
    const int64_t nG = 16;                      // materialised DW for kinds 1, 5 (16 x 4 MiB)
    float* G = (float*)rest;
    float* part = G + (size_t)nG * 1024 * 1024;  // split-K partial sums for kind 5 (2 Mi floats)
    char* rest2 = (char*)(part + (2 << 20));
    const size_t rest2_bytes = TDA_CALIBRATE_WS_BYTES - (size_t)(rest2 - base) - (1u << 20);
    // DW construction of a 2048 x 2048 layer at T = 512 (the same factor bytes viewed as 32
    // examples of 512 tokens): 4 DWs of 16 MiB
    tda_layer_desc L512 = L;
    L512.T = 512;
    L512.d_in = L512.d_out = 2048;
    const int64_t nB = 4;
    // Gram route on a 4096 x 4096 layer (the factor bytes viewed as 128 examples of 128 tokens)
    tda_layer_desc L4k = L;
    L4k.d_in = L4k.d_out = 4096;
    // Frobenius dots of 128 query and 128 train DWs of a 512 x 512 layer (1 MiB each): one
    // full query batch against one chunk of materialised train gradients
    const int64_t d5 = 512 * 512, nq5 = 128, nt5 = 128;
    float* G5 = (float*)rest2;
    const bool dots_tc = score_dots_tc(G5, nq5, d5, G5 + nq5 * d5, nt5, d5, d5);
    const int splits = score_splitk_splits(nq5, nt5, d5, dots_tc);
    if ((size_t)splits * nq5 * nt5 > ((size_t)2 << 20) || rest2_bytes < (size_t)(nq5 + nt5) * d5 * 4)
        return fail(TDA_ERR_WORKSPACE, "calibration scratch layout");
    for (int kind = 0; kind < kKinds; ++kind) {
        for (int rep = 0; rep < 4; ++rep) {
            if (rep == 1) cudaEventRecord(ev.a, s);
            if (kind == 0) {
                st = tda_project(&L, TDA_BF16, A, B, Nf, phi, 1024, TDA_ROUTE_FACTORED, nullptr, 0, s);
            } else if (kind == 1) {
                st = cuda_check(launch_materialize_G(L512, TDA_BF16, A, B, 0, nB, G, s), "calibrate DW");
            } else if (kind == 2) {
                st = tda_similarity_exact(&L4k, TDA_BF16, A, B, 8, A, B, 112, S, 112, 0.f, TDA_ROUTE_GRAM,
                                          nullptr, 0, s);
            } else if (kind == 3) {
                st = tda_similarity_projected(&L, TDA_BF16, A, B, 8, A, B, 64, S, 64, 0.f, TDA_ROUTE_GRAM, rest2,
                                              rest2_bytes, s);
            } else if (kind == 4) {
                st = tda_project(&L, TDA_BF16, A, B, 8, phi, 1024, TDA_ROUTE_MATERIALIZE, rest2, rest2_bytes, s);
            } else {
                st = cuda_check(
                    launch_score_splitk(G5, nq5, d5, G5 + nq5 * d5, nt5, d5, d5, S, nt5, 0.f, splits, part, dots_tc, s),
                    "calibrate dots");
            }
            if (st) return st;
        }
        cudaEventRecord(ev.b, s);
        if ((st = cuda_check(cudaEventSynchronize(ev.b), "calibration sync"))) return st;
        float ms = 0;
        cudaEventElapsedTime(&ms, ev.a, ev.b);
        secs[kind] = ms * 1e-3 / 3.0;
    }
    const double build = 2 * T * d * d;
    double rate[kKinds];
    rate[0] = Nf * (2 * T * (d * k + d * k) + 2 * T * k * k) / secs[0];
    rate[1] = nB * 2 * 512.0 * 2048.0 * 2048.0 / secs[1];
    rate[2] = 8 * 112 * 2 * T * T * (4096.0 + 4096.0) / secs[2];
    rate[3] = ((8 + 64) * 2 * T * (d * k + d * k) + 8 * 64 * 2 * T * T * (k + k)) / secs[3];
    // the projection's materialise route minus its construction (at T = 128): the sign projection alone
    const double sign_secs = secs[4] - 8 * build / rate[1];
    rate[4] = 8 * (2 * d * d * k + 2 * d * k * k) / (sign_secs > secs[4] * 0.05 ? sign_secs : secs[4] * 0.05);
    rate[5] = (double)nq5 * nt5 * 2 * d5 / secs[5];
    for (int r = 0; r < kKinds; ++r)
        if (!(rate[r] > 0) || !std::isfinite(rate[r])) rate[r] = 0;
    const double bw = secs[0] > 0 ? Nf * (T * (d + d) * 2 + 4 * k * k) / secs[0] : 0;
    set_route_rates(rate, bw);
    if (rates_out) {
        for (int r = 0; r < kKinds; ++r) rates_out[r] = rate[r];
        rates_out[kKinds] = bw;
    }
    return TDA_OK;
}
