// calibrate.cu -- device calibration of the route cost model (Sec. 3.2 and
// App. A.4 estimate costs per layer and op; on a given GPU the routes run at
// different rates, so the estimate becomes seconds = max(flops / rate_route,
// bytes / bandwidth) with rates measured here by short launches of the route
// kernels themselves).
#include "tda_internal.cuh"

namespace tda {
void set_route_rates(const double rate[4], double bw);
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
    double secs[4] = {0, 0, 0, 0};
    double flops[4] = {0, 0, 0, 0};
    double bytes_a = 0;
    for (int route = 0; route < 4; ++route) {
        for (int rep = 0; rep < 4; ++rep) {
            if (rep == 1) cudaEventRecord(ev.a, s);
            if (route == 0) {
                st = tda_project(&L, TDA_BF16, A, B, Nf, phi, 1024, TDA_ROUTE_FACTORED, nullptr, 0, s);
            } else if (route == 1) {
                st = tda_project(&L, TDA_BF16, A, B, 8, phi, 1024, TDA_ROUTE_MATERIALIZE, rest, rest_bytes, s);
            } else if (route == 2) {
                st = tda_similarity_exact(&L, TDA_BF16, A, B, 8, A, B, 256, S, 256, 0.f, TDA_ROUTE_GRAM,
                                          nullptr, 0, s);
            } else {  // Gram of projected (fp32) factors
                st = tda_similarity_projected(&L, TDA_BF16, A, B, 8, A, B, 64, S, 64, 0.f, TDA_ROUTE_GRAM, rest,
                                              rest_bytes, s);
            }
            if (st) return st;
        }
        cudaEventRecord(ev.b, s);
        if ((st = cuda_check(cudaEventSynchronize(ev.b), "calibration sync"))) return st;
        float ms = 0;
        cudaEventElapsedTime(&ms, ev.a, ev.b);
        secs[route] = ms * 1e-3 / 3.0;
    }
    const double T = 128, d = 1024, k = 32;
    flops[0] = Nf * (2 * T * (d * k + d * k) + 2 * T * k * k);
    flops[1] = 8 * (2 * T * d * d + 2 * d * d * k + 2 * d * k * k);
    flops[2] = 8 * 256 * 2 * T * T * (d + d);
    flops[3] = (8 + 64) * 2 * T * (d * k + d * k) + 8 * 64 * 2 * T * T * (k + k);
    bytes_a = Nf * (T * (d + d) * 2 + 4 * k * k);
    double rate[4];
    for (int r = 0; r < 4; ++r) rate[r] = secs[r] > 0 ? flops[r] / secs[r] : 0;
    const double bw = secs[0] > 0 ? bytes_a / secs[0] : 0;
    set_route_rates(rate, bw);
    if (rates_out) {
        rates_out[0] = rate[0];
        rates_out[1] = rate[1];
        rates_out[2] = rate[2];
        rates_out[3] = rate[3];
        rates_out[4] = bw;
    }
    return TDA_OK;
}
