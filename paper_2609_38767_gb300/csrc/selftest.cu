// selftest.cu -- tda_selftest_bounded_wait: exercises the bounded-wait path the
// tensor-core kernels rely on. One CTA initialises an mbarrier that nothing
// ever arrives on and waits on it with the same bounded loop (%globaltimer
// limit); on expiry it ORs kErrTimeout into the library's device error word and
// returns normally, so the context stays usable.
#include "tda_internal.cuh"

namespace tda {
namespace {

__global__ void bounded_wait_kernel(uint64_t timeout_ns, unsigned int* err) {
    __shared__ __align__(8) uint64_t bar;
    const uint32_t b = (uint32_t)__cvta_generic_to_shared(&bar);
    asm volatile("mbarrier.init.shared::cta.b64 [%0], 1;" ::"r"(b) : "memory");
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    uint64_t t0;
    asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t0));
    while (true) {
        uint32_t ok;
        asm volatile(
            "{\n .reg .pred p;\n mbarrier.try_wait.parity.shared::cta.b64 p, [%1], 0;\n selp.u32 %0, 1, 0, p;\n}"
            : "=r"(ok)
            : "r"(b)
            : "memory");
        if (ok) return;  // never: no thread arrives
        uint64_t t;
        asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
        if (t - t0 > timeout_ns) {
            atomicOr(err, kErrTimeout);
            return;
        }
    }
}

}  // namespace
}  // namespace tda

using namespace tda;

extern "C" tda_status tda_selftest_bounded_wait(uint64_t timeout_ns, void* stream) {
    if (timeout_ns == 0 || timeout_ns > 2000000000ull)
        return fail(TDA_ERR_INVALID_ARG, "timeout_ns must be in (0, 2e9]");
    unsigned int* err = device_error_word();
    if (!err) return fail(TDA_ERR_CUDA, "cannot resolve the device error word");
    note_launches(1);
    bounded_wait_kernel<<<1, 1, 0, (cudaStream_t)stream>>>(timeout_ns, err);
    return cuda_check(cudaGetLastError(), "selftest launch");
}
