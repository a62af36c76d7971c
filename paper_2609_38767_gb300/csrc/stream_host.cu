// stream_host.cu -- tda_project_host: the factored projection of factors that
// live in host memory. App. A.2 applies the projection as the factors arrive,
// so raw factors are never buffered whole; here they stream through two
// device staging halves of the caller's scratch: the copies of chunk c+1
// overlap the projection of chunk c (on the caller's stream). Each chunk's
// bytes are split evenly over kCopyStreams library-owned copy streams: on the
// GB300 machines measured, one stream moved 106-135 GB/s host to device and
// three concurrent ones up to 183 GB/s.
#include <mutex>

#include "tda_internal.cuh"

namespace tda {
namespace {

constexpr int kCopyStreams = 4;

struct HostPipe {
    bool ready = false;
    cudaStream_t copy[kCopyStreams] = {};
    cudaEvent_t copied[2][kCopyStreams] = {};  // [half][stream]
    cudaEvent_t done[2] = {nullptr, nullptr};
    uint64_t next = 0;  // staging half of the next chunk: alternates across calls too
    std::mutex mu;
};

HostPipe g_pipes[64];

cudaError_t pipe_for_device(HostPipe** out) {
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    if (dev < 0 || dev >= 64) return cudaErrorInvalidDevice;
    HostPipe& p = g_pipes[dev];
    *out = &p;
    if (p.ready) return cudaSuccess;
    for (int i = 0; i < kCopyStreams; ++i)
        if ((e = cudaStreamCreateWithFlags(&p.copy[i], cudaStreamNonBlocking)) != cudaSuccess) return e;
    for (int b = 0; b < 2; ++b) {
        for (int i = 0; i < kCopyStreams; ++i)
            if ((e = cudaEventCreateWithFlags(&p.copied[b][i], cudaEventDisableTiming)) != cudaSuccess) return e;
        if ((e = cudaEventCreateWithFlags(&p.done[b], cudaEventDisableTiming)) != cudaSuccess) return e;
    }
    p.ready = true;
    return cudaSuccess;
}

}  // namespace
}  // namespace tda

using namespace tda;

extern "C" size_t tda_project_host_ws_min(const tda_layer_desc* L, tda_dtype dtype) {
    if (!L || L->T < 0 || L->d_in < 1 || L->d_out < 1) return 0;
    const size_t el = dtype == TDA_F32 ? 4 : 2;
    const size_t per = (size_t)L->T * (size_t)(L->d_in + L->d_out) * el;
    return 2 * (((per + 255) / 256) * 256);
}

extern "C" tda_status tda_project_host(const tda_layer_desc* L, tda_dtype dtype, const void* A_h,
                                       const void* B_h, int64_t N, float* phi, int64_t ld_phi,
                                       void* ws, size_t ws_bytes, void* stream) {
    if (!L) return fail(TDA_ERR_INVALID_ARG, "layer descriptor is NULL");
    if (dtype != TDA_F32 && dtype != TDA_BF16) return fail(TDA_ERR_INVALID_ARG, "dtype must be F32 or BF16");
    if (N < 0) return fail(TDA_ERR_INVALID_ARG, "negative N");
    if (N > 0 && L->T > 0 && (!A_h || !B_h)) return fail(TDA_ERR_INVALID_ARG, "NULL host factor pointer");
    const size_t need = tda_project_host_ws_min(L, dtype);
    if (need == 0) return fail(TDA_ERR_INVALID_ARG, "bad layer sizes");
    if (!ws || ws_bytes < need)
        return fail(TDA_ERR_WORKSPACE, "tda_project_host needs >= %zu bytes of ws, got %zu", need, ws_bytes);
    if ((uintptr_t)ws & 255) return fail(TDA_ERR_INVALID_ARG, "ws must be 256-byte aligned");
    if (N == 0 || L->T == 0)
        return tda_project(L, dtype, ws, ws, N, phi, ld_phi, TDA_ROUTE_FACTORED, nullptr, 0, stream);

    HostPipe* p = nullptr;
    tda_status st = cuda_check(pipe_for_device(&p), "copy pipeline setup");
    if (st) return st;
    std::lock_guard<std::mutex> lock(p->mu);
    const size_t el = dtype == TDA_F32 ? 4 : 2;
    const size_t a_ex = (size_t)L->T * L->d_in * el, b_ex = (size_t)L->T * L->d_out * el;
    // Room beyond the minimum: the projection's own optional workspace, one per staging half
    // (its uses are ordered by the same events as the half's), taken from the end of ws.
    size_t pws = 0;
    if (tda_workspace_size(TDA_OP_PROJECT, L, dtype, 1, 0, TDA_ROUTE_FACTORED, &pws) != TDA_OK) pws = 0;
    pws = (pws + 255) & ~(size_t)255;
    if (pws && ws_bytes < need + 2 * pws) pws = 0;
    // Staging halves of at most ~2.4 GB (at least one example each): on a GB300, calls whose
    // halves were 4.8 GB apart sustained ~120 GB/s against ~210 GB/s with 2.4 GB halves.
    const size_t half0 = ((ws_bytes - 2 * pws) / 2) & ~(size_t)255;  // the projection workspaces follow 2 * half0
    size_t half = half0;
    const size_t half_cap = ((size_t)2400 << 20) > ((a_ex + b_ex + 255) & ~(size_t)255)
                                ? ((size_t)2400 << 20)
                                : ((a_ex + b_ex + 255) & ~(size_t)255);
    if (half > half_cap) half = half_cap;
    int64_t chunk = (int64_t)(half / (a_ex + b_ex));
    if (chunk > N) chunk = N;

    cudaStream_t s = (cudaStream_t)stream;
    for (int64_t c0 = 0; c0 < N; c0 += chunk) {
        // consecutive chunks, also of consecutive calls, use alternate halves: the copy of the
        // next one overlaps the projection of this one (done[] orders reuse of a half)
        const int b = (int)(p->next++ & 1);
        const int64_t cnt = (N - c0) < chunk ? (N - c0) : chunk;
        char* dA = (char*)ws + (size_t)b * half;
        char* dB = dA + (size_t)chunk * a_ex;
        const char* srcA = (const char*)A_h + (size_t)c0 * a_ex;
        const char* srcB = (const char*)B_h + (size_t)c0 * b_ex;
        const size_t nA = (size_t)cnt * a_ex, nB = (size_t)cnt * b_ex;
        for (int i = 0; i < kCopyStreams; ++i) {
            // part i of each factor: bytes [i n / kCopyStreams, (i + 1) n / kCopyStreams), 256-byte cuts
            auto cut = [](size_t n, int k) {
                const size_t c = ((n * (size_t)k / kCopyStreams) + 255) & ~(size_t)255;
                return c < n ? c : n;
            };
            const size_t a0 = i == 0 ? 0 : cut(nA, i), a1 = i + 1 == kCopyStreams ? nA : cut(nA, i + 1);
            const size_t b0 = i == 0 ? 0 : cut(nB, i), b1 = i + 1 == kCopyStreams ? nB : cut(nB, i + 1);
            if ((st = cuda_check(cudaStreamWaitEvent(p->copy[i], p->done[b], 0), "wait buffer"))) return st;
            if (a1 > a0 && (st = cuda_check(cudaMemcpyAsync(dA + a0, srcA + a0, a1 - a0, cudaMemcpyHostToDevice,
                                                            p->copy[i]),
                                            "copy A")))
                return st;
            if (b1 > b0 && (st = cuda_check(cudaMemcpyAsync(dB + b0, srcB + b0, b1 - b0, cudaMemcpyHostToDevice,
                                                            p->copy[i]),
                                            "copy B")))
                return st;
            if ((st = cuda_check(cudaEventRecord(p->copied[b][i], p->copy[i]), "record copy"))) return st;
            if ((st = cuda_check(cudaStreamWaitEvent(s, p->copied[b][i], 0), "wait copy"))) return st;
        }
        void* pw = pws ? (char*)ws + 2 * half0 + (size_t)b * pws : nullptr;
        if ((st = tda_project(L, dtype, dA, dB, cnt, phi + c0 * ld_phi, ld_phi, TDA_ROUTE_FACTORED, pw, pws,
                              stream)))
            return st;
        if ((st = cuda_check(cudaEventRecord(p->done[b], s), "record done"))) return st;
    }
    return TDA_OK;
}
