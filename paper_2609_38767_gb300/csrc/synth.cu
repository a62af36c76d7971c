// synth.cu -- device implementation of the seeded synthetic-factor generator
// (libtda_synth.so). The definition, and the bit-identical numpy version,
// are in paper_2609_38767_gb300/synth.py. Every floating-point operation is
// written with an explicit rounding intrinsic so that the compiler cannot
// contract it and the result matches one-rounding-per-operation IEEE fp32.
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "../../include/tda_synth.h"

namespace {

constexpr uint64_t kG = 0x9E3779B97F4A7C15ull;

__host__ __device__ __forceinline__ uint64_t smix(uint64_t z) {
    z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
    z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
    return z ^ (z >> 31);
}

__device__ __forceinline__ uint64_t sword(uint64_t key, uint64_t n) { return smix(key + kG * (n + 1u)); }

__device__ __forceinline__ float snormal(uint64_t key, uint64_t i) {
    int64_t s = 0;
#pragma unroll
    for (int j = 0; j < 3; ++j) {
        const uint64_t w = sword(key, 3u * i + (uint64_t)j);
        s += (int64_t)(w & 0xFFFFu) + (int64_t)((w >> 16) & 0xFFFFu) + (int64_t)((w >> 32) & 0xFFFFu) +
             (int64_t)((w >> 48) & 0xFFFFu);
    }
    return __fdiv_rn((float)(s + 6 - 393216), 65536.0f);
}

__device__ __forceinline__ float sstudent4(uint64_t key, uint64_t i) {
    const uint64_t b = 5u * i;
    const float z0 = snormal(key, b), z1 = snormal(key, b + 1), z2 = snormal(key, b + 2),
                z3 = snormal(key, b + 3), z4 = snormal(key, b + 4);
    float s = __fmul_rn(z1, z1);
    s = __fadd_rn(s, __fmul_rn(z2, z2));
    s = __fadd_rn(s, __fmul_rn(z3, z3));
    s = __fadd_rn(s, __fmul_rn(z4, z4));
    s = __fmul_rn(s, 0.25f);
    return s > 0.f ? __fdiv_rn(z0, __fsqrt_rn(s)) : 0.f;
}

template <typename T>
__device__ __forceinline__ void store(T* p, float v);
template <>
__device__ __forceinline__ void store<float>(float* p, float v) { *p = v; }
template <>
__device__ __forceinline__ void store<__nv_bfloat16>(__nv_bfloat16* p, float v) { *p = __float2bfloat16_rn(v); }

template <typename T>
__global__ void fill_kernel(T* __restrict__ X, int dist, uint64_t key, int64_t e0, int64_t n, int64_t Tn,
                            int64_t d, float sigma, uint64_t mkey, uint64_t mthr) {
    const int64_t total = n * Tn * d;
    for (int64_t e = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; e < total;
         e += (int64_t)gridDim.x * blockDim.x) {
        const int64_t ex = e / (Tn * d);
        const int64_t rem = e - ex * Tn * d;
        const int64_t t = rem / d;
        const uint64_t tok = (uint64_t)(e0 + ex) * (uint64_t)Tn + (uint64_t)t;
        const uint64_t i = tok * (uint64_t)d + (uint64_t)(rem - t * d);
        float v = 0.f;
        if (mthr == 0 || sword(mkey, tok) >= mthr) {
            v = dist == 0 ? snormal(key, i) : sstudent4(key, i);
            v = __fmul_rn(v, sigma);
        }
        store<T>(X + e, v);
    }
}

}  // namespace

extern "C" int32_t tda_synth_fill(void* X, int32_t dtype, int32_t dist, uint64_t seed, uint64_t stream_id,
                                  int64_t e0, int64_t n, int64_t T, int64_t d, float sigma,
                                  uint64_t mask_seed, uint64_t mask_stream, uint64_t mask_threshold,
                                  void* stream) {
    if ((dtype != 0 && dtype != 1) || (dist != 0 && dist != 1) || n < 0 || T < 0 || d < 0 || e0 < 0) return 1;
    if (n * T * d == 0) return 0;
    if (!X) return 1;
    const uint64_t key = smix(seed + kG * (stream_id + 1u));
    const uint64_t mkey = smix(mask_seed + kG * (mask_stream + 1u));
    const int64_t total = n * T * d;
    int64_t blocks = (total + 255) / 256;
    if (blocks > 152 * 32) blocks = 152 * 32;
    cudaStream_t s = (cudaStream_t)stream;
    if (dtype == 1)
        fill_kernel<__nv_bfloat16><<<(unsigned)blocks, 256, 0, s>>>((__nv_bfloat16*)X, dist, key, e0, n, T, d,
                                                                    sigma, mkey, mask_threshold);
    else
        fill_kernel<float><<<(unsigned)blocks, 256, 0, s>>>((float*)X, dist, key, e0, n, T, d, sigma, mkey,
                                                            mask_threshold);
    return cudaGetLastError() == cudaSuccess ? 0 : 2;
}
