// k_materialize_tc.cu -- route (b)'s materialisation DW = g a^T (Eq. 1),
// G[r][c] = sum_t B[t][r] A[t][c], on the tcgen05 tensor cores for bf16
// factors: M = 128 rows of d_out, N = 256 columns of d_in, K = the tokens.
//
// Both MMA operands need the token axis contiguous (K-major), but in memory a
// token's features are contiguous, so producer warps transpose 64-token slabs
// on the way into shared memory: each thread loads two 16-byte runs of 8
// features from consecutive tokens t, t+1 and writes eight (t, t+1) bf16 pairs
// into the 128-byte-swizzled K-major operand layout. The MMA warp accumulates
// a 128 x 256 fp32 tile in TMEM (double-buffered), the epilogue warps stream it
// to G.
//
// Warp roles (288 threads): warps 0-3 transposing producers, warp 4 TMEM
// allocator and MMA issuer (lane 0), warps 5-8 epilogue (one TMEM lane
// quadrant each). Waits are bounded (about 1 s) and set kErrTimeout on expiry.
#include <cuda.h>
#include <cuda_bf16.h>

#include "tda_internal.cuh"

namespace tda {
namespace {

#include "tc_ptx.cuh"

constexpr int kThreads = 288;
constexpr int kTM = 128, kTN = 256, kTK = 64;       // tile rows (d_out), columns (d_in), tokens per stage
constexpr uint32_t kABytes = kTM * kTK * 2;         // 16 KiB
constexpr uint32_t kBBytes = kTN * kTK * 2;         // 32 KiB
constexpr uint32_t kStageBytes = kABytes + kBBytes;
constexpr int kStages = 4;
constexpr uint32_t kTmemCols = 512;                 // two 128 x 256 fp32 accumulators
constexpr size_t kSmem = 1024 + (size_t)kStages * kStageBytes + 8 * (2 * kStages + 5) + 16;
static_assert(kSmem <= 232448, "shared memory per CTA");

struct MParams {
    const __nv_bfloat16* A;  // [.][T][d_in]
    const __nv_bfloat16* B;  // [.][T][d_out]
    float* G;                // [n][d_out][d_in]
    int64_t n, T, d_in, d_out;
    int64_t n_rb, n_cb, n_units;
    unsigned int* err;
};

// Byte offset of element (row m, k) in a K-major, 128-byte-swizzled bf16 tile.
__device__ __forceinline__ uint32_t sw_off(int m, int k) {
    const int kb = k * 2;
    return (uint32_t)((m >> 3) * 1024 + (m & 7) * 128 + ((((kb >> 4) ^ (m & 7))) << 4) + (kb & 15));
}

// Transpose a 64-token slab of X (rows t0.., features f0.. f0+rows-1) into a
// K-major tile of `rows` operand rows: operand row m, k = token offset.
__device__ __forceinline__ void fill_tile(uint8_t* tile, const __nv_bfloat16* X, int64_t T, int64_t d, int64_t t0,
                                          int64_t f0, int rows, int tid) {
    const int groups = rows / 8;  // 8-feature runs per token
    for (int u = tid; u < groups * (kTK / 2); u += 128) {
        // a warp covers the 32 token pairs of one feature run: its eight stores per
        // step then land on 32 distinct words of one 128-byte operand row (no bank conflicts)
        const int kp = u % (kTK / 2), g = u / (kTK / 2);
        const int m0 = g * 8, k = kp * 2;
        const int64_t t = t0 + k, f = f0 + m0;
        uint4 v0 = make_uint4(0, 0, 0, 0), v1 = v0;
        if (f + 8 <= d) {
            if (t < T) v0 = *reinterpret_cast<const uint4*>(X + t * d + f);
            if (t + 1 < T) v1 = *reinterpret_cast<const uint4*>(X + (t + 1) * d + f);
        } else if (f < d) {  // ragged feature tail (d % 8 == 0 makes this unreachable for whole runs)
            const uint16_t* x0 = reinterpret_cast<const uint16_t*>(X + t * d);
            uint16_t a[8] = {}, b[8] = {};
            for (int j = 0; j < 8 && f + j < d; ++j) {
                if (t < T) a[j] = x0[f + j];
                if (t + 1 < T) b[j] = x0[d + f + j];
            }
            v0 = make_uint4(a[0] | (a[1] << 16), a[2] | (a[3] << 16), a[4] | (a[5] << 16), a[6] | (a[7] << 16));
            v1 = make_uint4(b[0] | (b[1] << 16), b[2] | (b[3] << 16), b[4] | (b[5] << 16), b[6] | (b[7] << 16));
        }
        const uint32_t w0[4] = {v0.x, v0.y, v0.z, v0.w}, w1[4] = {v1.x, v1.y, v1.z, v1.w};
#pragma unroll
        for (int j = 0; j < 8; ++j) {
            const uint32_t lo = (w0[j >> 1] >> (16 * (j & 1))) & 0xFFFFu;
            const uint32_t hi = (w1[j >> 1] >> (16 * (j & 1))) & 0xFFFFu;
            *reinterpret_cast<uint32_t*>(tile + sw_off(m0 + j, k)) = lo | (hi << 16);
        }
    }
}

__global__ void __launch_bounds__(kThreads, 1) materialize_tc_kernel(const MParams p) {
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = (uint8_t*)(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
    uint64_t* bars = (uint64_t*)(smem + (size_t)kStages * kStageBytes);
    uint64_t* full = bars;                  // producers wrote the stage (count 4)
    uint64_t* empty = bars + kStages;       // MMAs done with the stage (count 1)
    uint64_t* tfull = bars + 2 * kStages;   // [2] accumulator ready
    uint64_t* tempty = tfull + 2;           // [2] accumulator drained (count 4)
    uint64_t* mma_done = tempty + 2;
    uint32_t* tmem_slot = (uint32_t*)(mma_done + 1);
    volatile int* abort = (volatile int*)(tmem_slot + 1);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    if (threadIdx.x == 0) {
        for (int s = 0; s < kStages; ++s) {
            mbar_init(smem_u32(&full[s]), 4);
            mbar_init(smem_u32(&empty[s]), 1);
        }
        for (int b = 0; b < 2; ++b) {
            mbar_init(smem_u32(&tfull[b]), 1);
            mbar_init(smem_u32(&tempty[b]), 4);
        }
        mbar_init(smem_u32(mma_done), 1);
        *abort = 0;
        fence_mbar_init();
    }
    if (warp == 4) {
        tmem_alloc(smem_u32(tmem_slot), kTmemCols);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *tmem_slot;
    const int nk = (int)((p.T + kTK - 1) / kTK);

    if (warp < 4) {
        // ---------------- transposing producers
        uint32_t ring = 0;
        bool ok = true;
        for (int64_t u = blockIdx.x; ok && u < p.n_units; u += gridDim.x) {
            const int64_t e = u / (p.n_rb * p.n_cb), rc = u % (p.n_rb * p.n_cb);
            const int64_t r0 = (rc / p.n_cb) * kTM, c0 = (rc % p.n_cb) * kTN;
            const __nv_bfloat16* Be = p.B + e * p.T * p.d_out;
            const __nv_bfloat16* Ae = p.A + e * p.T * p.d_in;
            for (int kc = 0; kc < nk; ++kc, ++ring) {
                const int s = ring % kStages;
                const uint32_t ph = (ring / kStages) & 1u;
                bool got = true;
                if (lane == 0) got = wait_bounded(smem_u32(&empty[s]), ph ^ 1u, abort, p.err);
                got = __shfl_sync(0xffffffffu, got, 0);
                if (!got) {
                    ok = false;
                    break;
                }
                uint8_t* st = smem + (size_t)s * kStageBytes;
                fill_tile(st, Be, p.T, p.d_out, (int64_t)kc * kTK, r0, kTM, threadIdx.x);
                fill_tile(st + kABytes, Ae, p.T, p.d_in, (int64_t)kc * kTK, c0, kTN, threadIdx.x);
                fence_proxy_async();
                __syncwarp();
                if (lane == 0) mbar_arrive(smem_u32(&full[s]));
            }
        }
    } else if (warp == 4) {
        if (lane == 0) {
            // ---------------- MMA issuer
            uint32_t ring = 0, tile = 0;
            bool ok = true;
            const uint32_t idesc = idesc_bf16(kTM, kTN);
            for (int64_t u = blockIdx.x; ok && u < p.n_units; u += gridDim.x, ++tile) {
                const uint32_t b = tile & 1u, use = tile >> 1;
                if (!wait_bounded(smem_u32(&tempty[b]), (use & 1u) ^ 1u, abort, p.err)) break;
                tc_fence_after();
                for (int kc = 0; kc < nk; ++kc, ++ring) {
                    const int s = ring % kStages;
                    const uint32_t ph = (ring / kStages) & 1u;
                    if (!wait_bounded(smem_u32(&full[s]), ph, abort, p.err)) {
                        ok = false;
                        break;
                    }
                    tc_fence_after();
                    uint8_t* st = smem + (size_t)s * kStageBytes;
                    const uint64_t ad = sw128_desc(smem_u32(st)), bd = sw128_desc(smem_u32(st + kABytes));
#pragma unroll
                    for (int k = 0; k < kTK / 16; ++k)
                        mma_bf16(tmem + b * kTN, ad + 2 * k, bd + 2 * k, idesc, (kc > 0 || k > 0) ? 1u : 0u);
                    mma_commit(smem_u32(&empty[s]));
                }
                if (!ok) break;
                mma_commit(smem_u32(&tfull[b]));
            }
            mma_commit(smem_u32(mma_done));
            const uint64_t t0 = global_ns();
            while (!mbar_try_wait(smem_u32(mma_done), 0))
                if (global_ns() - t0 > kTimeoutNs) {
                    atomicOr(p.err, kErrTimeout);
                    break;
                }
        }
    } else {
        // ---------------- epilogue: TMEM -> G
        const int q = warp & 3, row = q * 32 + lane;
        uint32_t tile = 0;
        for (int64_t u = blockIdx.x; u < p.n_units; u += gridDim.x, ++tile) {
            const uint32_t b = tile & 1u, use = tile >> 1;
            bool got = true;
            if (lane == 0) got = wait_bounded(smem_u32(&tfull[b]), use & 1u, abort, p.err);
            got = __shfl_sync(0xffffffffu, got, 0);
            if (epi_any(!got)) break;
            tc_fence_after();
            const int64_t e = u / (p.n_rb * p.n_cb), rc = u % (p.n_rb * p.n_cb);
            const int64_t r = (rc / p.n_cb) * kTM + row, c0 = (rc % p.n_cb) * kTN;
            float* gr = p.G + (e * p.d_out + r) * p.d_in;
            const uint32_t tb = tmem + ((uint32_t)(q * 32) << 16) + b * kTN;
#pragma unroll 4
            for (int c = 0; c < kTN; c += 16) {
                float v[16];
                tmem_ld16(tb + c, v);
                if (r < p.d_out) {
                    const int64_t cc = c0 + c;
                    if (cc + 16 <= p.d_in) {
#pragma unroll
                        for (int i = 0; i < 16; i += 4)
                            *reinterpret_cast<float4*>(gr + cc + i) = make_float4(v[i], v[i + 1], v[i + 2], v[i + 3]);
                    } else {
                        for (int i = 0; i < 16 && cc + i < p.d_in; ++i) gr[cc + i] = v[i];
                    }
                }
            }
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(smem_u32(&tempty[b]));
        }
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 4) {
        tc_fence_after();
        tmem_dealloc(tmem, kTmemCols);
    }
}

}  // namespace

bool materialize_tc_supported(const tda_layer_desc& L, tda_dtype dt, const void* A, const void* B, const float* G) {
    static int sm103 = -1;
    if (sm103 < 0) {
        int dev = 0, major = 0, minor = 0;
        cudaGetDevice(&dev);
        cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev);
        cudaDeviceGetAttribute(&minor, cudaDevAttrComputeCapabilityMinor, dev);
        sm103 = (major == 10 && minor == 3) ? 1 : 0;
    }
    return sm103 && dt == TDA_BF16 && L.T >= 1 && L.d_in % 8 == 0 && L.d_out % 8 == 0 && L.d_in % 4 == 0 &&
           ((uintptr_t)A & 15) == 0 && ((uintptr_t)B & 15) == 0 && ((uintptr_t)G & 15) == 0;
}

// G[i][r][c] (i < n) of examples e0 .. e0+n-1 of bf16 factors A, B.
cudaError_t launch_materialize_tc(const tda_layer_desc& L, const void* A, const void* B, int64_t e0, int64_t n,
                                  float* G, unsigned int* err, cudaStream_t s) {
    if (n == 0) return cudaSuccess;
    MParams p;
    p.A = (const __nv_bfloat16*)A + e0 * L.T * L.d_in;
    p.B = (const __nv_bfloat16*)B + e0 * L.T * L.d_out;
    p.G = G;
    p.n = n;
    p.T = L.T;
    p.d_in = L.d_in;
    p.d_out = L.d_out;
    p.n_rb = (L.d_out + kTM - 1) / kTM;
    p.n_cb = (L.d_in + kTN - 1) / kTN;
    p.n_units = n * p.n_rb * p.n_cb;
    p.err = err;
    static int sms = 0;
    if (!sms) {
        int dev = 0;
        cudaGetDevice(&dev);
        cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
        if (sms <= 0) sms = 1;
    }
    cudaError_t e = cudaFuncSetAttribute(materialize_tc_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kSmem);
    if (e != cudaSuccess) return e;
    const int64_t grid = p.n_units < sms ? p.n_units : sms;
    note_launches(1);
    materialize_tc_kernel<<<(unsigned)grid, kThreads, kSmem, s>>>(p);
    return cudaGetLastError();
}

}  // namespace tda
