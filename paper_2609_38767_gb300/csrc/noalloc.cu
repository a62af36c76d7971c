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
#include <cuda.h>

#include <mutex>

#include "tda_internal.cuh"

namespace tda {
namespace {

constexpr size_t kNoAllocScratchBytes = (size_t)64 << 20;  // 64 MiB

// The shared scratch. In host code this name is only a host-side stand-in for
// the symbol, never a device address: the address is resolved per CUDA
// context with cudaGetSymbolAddress below.
static __device__ __align__(256) unsigned char g_noalloc_scratch[kNoAllocScratchBytes];

typedef CUresult (*CtxGetCurrentFn)(CUcontext*);

CtxGetCurrentFn ctx_get_current() {
    static CtxGetCurrentFn fn = nullptr;
    static std::once_flag once;
    std::call_once(once, [] {
        void* f = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuCtxGetCurrent", &f, 12000, cudaEnableDefault, &q) == cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = (CtxGetCurrentFn)f;
    });
    return fn;
}

// Resolved addresses, one per CUDA context (the array lives in each context
// that loads this module: normally the runtime's primary context of a device).
struct Slot {
    CUcontext ctx;
    void* ptr;
};
std::mutex g_noalloc_mu;
Slot g_noalloc_slots[64] = {};
int g_noalloc_nslots = 0;

// The first call in a context resolves the array's device address (with lazy
// module loading that call also loads the module, which commits the 64 MiB);
// later calls in the same context reuse it.
cudaError_t noalloc_scratch(void** out) {
    CtxGetCurrentFn get = ctx_get_current();
    if (!get) return cudaErrorNotSupported;
    std::lock_guard<std::mutex> lock(g_noalloc_mu);
    CUcontext ctx = nullptr;
    if (get(&ctx) != CUDA_SUCCESS) return cudaErrorUnknown;
    for (int i = 0; ctx && i < g_noalloc_nslots; ++i)
        if (g_noalloc_slots[i].ctx == ctx) {
            *out = g_noalloc_slots[i].ptr;
            return cudaSuccess;
        }
    void* p = nullptr;
    cudaError_t e = cudaGetSymbolAddress(&p, g_noalloc_scratch);  // binds the primary context if none is current
    if (e != cudaSuccess) return e;
    if (!ctx && get(&ctx) != CUDA_SUCCESS) return cudaErrorUnknown;
    if (g_noalloc_nslots < 64) g_noalloc_slots[g_noalloc_nslots++] = Slot{ctx, p};
    *out = p;
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
