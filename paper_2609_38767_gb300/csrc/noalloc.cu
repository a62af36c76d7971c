// noalloc.cu -- tda_project_materialized_noalloc: the materialise-route
// projection with its scratch in a fixed device array owned by this library
// instead of a caller-supplied workspace.
//
// Who needs it: callers that cannot call cudaMalloc (or hand out a scratch
// buffer) at the point where they project gradients -- for example a plugin
// running inside a host program that owns and partitions all device memory
// itself, or a latency-critical loop that must not pay cudaMalloc's implicit
// device-wide synchronisation. They still pass their own inputs and outputs.
//
// Cost of the convenience: every GPU that loads libtda.so holds the array
// (kNoAllocScratchBytes) from module load until process exit, and all calls
// share it.
#include <mutex>

#include "tda_internal.cuh"

namespace tda {
namespace {

constexpr size_t kNoAllocScratchBytes = (size_t)64 << 20;  // 64 MiB

// The shared scratch. In host code this name is only a host-side stand-in for
// the symbol, never a device address: the address is resolved per device with
// cudaGetSymbolAddress below.
static __device__ __align__(256) unsigned char g_noalloc_scratch[kNoAllocScratchBytes];

std::mutex g_noalloc_mu;
void* g_noalloc_ptr[64] = {};

// First call on a device (with that device current) resolves the array's
// device address; later calls reuse it.
cudaError_t noalloc_scratch(void** out) {
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    if (dev < 0 || dev >= 64) return cudaErrorInvalidDevice;
    std::lock_guard<std::mutex> lock(g_noalloc_mu);
    if (!g_noalloc_ptr[dev]) {
        void* p = nullptr;
        e = cudaGetSymbolAddress(&p, g_noalloc_scratch);
        if (e != cudaSuccess) return e;
        g_noalloc_ptr[dev] = p;
    }
    *out = g_noalloc_ptr[dev];
    return cudaSuccess;
}

}  // namespace
}  // namespace tda

using namespace tda;

extern "C" size_t tda_noalloc_scratch_bytes(void) { return kNoAllocScratchBytes; }

extern "C" tda_status tda_project_materialized_noalloc(const tda_layer_desc* L, tda_dtype dtype, const void* A,
                                                       const void* B, int64_t N, float* phi, int64_t ld_phi,
                                                       void* stream) {
    if (!L) return fail(TDA_ERR_INVALID_ARG, "layer descriptor is NULL");
    if (L->d_in < 1 || L->d_out < 1 || L->T < 0 || L->k_in < 1 || L->k_out < 1)
        return fail(TDA_ERR_INVALID_ARG, "bad layer sizes");
    const size_t need = materialize_ws_bytes_per_example(*L);
    if (need > kNoAllocScratchBytes)
        return fail(TDA_ERR_WORKSPACE,
                    "layer needs %zu bytes of scratch per example (d_out*d_in + d_out*k_in floats); the "
                    "built-in scratch holds %zu bytes -- use tda_project with a caller workspace",
                    need, kNoAllocScratchBytes);
    void* scratch = nullptr;
    if (N > 0 && L->T > 0) {
        tda_status st = cuda_check(noalloc_scratch(&scratch), "resolve built-in scratch");
        if (st) return st;
    }
    // The materialise kernels overwrite every scratch element they later read,
    // so the previous call's contents need no clearing.
    return tda_project(L, dtype, A, B, N, phi, ld_phi, TDA_ROUTE_MATERIALIZE, scratch,
                       scratch ? kNoAllocScratchBytes : 0, stream);
}
