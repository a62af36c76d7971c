// k_materialize_tc.cu -- route (b)'s materialisation DW = g a^T (Eq. 1),
// G[r][c] = sum_t B[t][r] A[t][c], on the tcgen05 tensor cores for bf16
// factors: M = 128 rows of d_out, N = 256 columns of d_in, K = the tokens.
//
// The contraction runs over tokens, and in memory a token's features are
// contiguous, so both operands are MN-major: TMA copies 64-feature x 64-token
// boxes (128-byte swizzle) straight into the canonical MN-major layout, where
// a swizzle atom is 64 features x 8 tokens (1 KiB), the 8-token groups follow
// each other 1 KiB apart (SBO) and the 64-feature atoms of one operand sit one
// box (8 KiB) apart (LBO). Tokens past T and features past d arrive as zeros
// (3-D tensor map over [n][T][d]). The MMA warp accumulates a 128 x 256 fp32
// tile in TMEM (double-buffered); each epilogue warp stages 32 x 32 blocks of
// it in shared memory (two buffers) and TMA stores them to G, clipped at the
// matrix edges.
//
// Warp roles (192 threads): warp 0 TMA producer (lane 0), warp 1 TMEM
// allocator and MMA issuer (lane 0), warps 2-5 epilogue (TMEM lane quadrant
// warp % 4). Waits are bounded (about 1 s) and set kErrTimeout on expiry.
#include <cuda.h>
#include <cuda_bf16.h>

#include <mutex>

#include "tda_internal.cuh"

namespace tda {
namespace {

#include "tc_ptx.cuh"

constexpr int kThreads = 192;
constexpr int kTM = 128, kTN = 256, kTK = 64;       // tile rows (d_out), columns (d_in), tokens per stage
constexpr uint32_t kBox = 64 * kTK * 2;             // one 64-feature x 64-token box: 8 KiB
constexpr uint32_t kABytes = kTM * kTK * 2;         // 16 KiB (2 boxes)
constexpr uint32_t kBBytes = kTN * kTK * 2;         // 32 KiB (4 boxes)
constexpr uint32_t kStageBytes = kABytes + kBBytes;
constexpr int kStages = 4;
constexpr uint32_t kTmemCols = 512;                 // two 128 x 256 fp32 accumulators
constexpr uint32_t kOutBox = 32 * 32 * 4;            // one 32 x 32 fp32 block of G (128-byte swizzled rows)
constexpr uint32_t kOutBytes = 4 * 2 * kOutBox;      // two blocks per epilogue warp
constexpr size_t kSmem = 1024 + (size_t)kStages * kStageBytes + kOutBytes + 8 * (2 * kStages + 5) + 16;
static_assert(kSmem <= 232448, "shared memory per CTA");

struct MParams {
    float* G;  // [n][d_out][d_in]
    int64_t n, d_in, d_out;
    int64_t n_rb, n_cb, n_units;
    int nk;    // token chunks of kTK
    unsigned int* err;
};

// Shared-memory matrix descriptor for an MN-major, 128-byte-swizzled bf16
// operand: LBO = distance between 64-element MN atoms, SBO = distance between
// 8-row K groups (both in bytes, multiples of 16), tile base 1024-byte aligned.
__device__ __forceinline__ uint64_t sw128_mn_desc(uint32_t saddr, uint32_t lbo, uint32_t sbo) {
    return (uint64_t)((saddr & 0x3FFFFu) >> 4) | ((uint64_t)(lbo >> 4) << 16) | ((uint64_t)(sbo >> 4) << 32) |
           ((uint64_t)1 << 46) | ((uint64_t)2 << 61);
}
// kind::f16 instruction descriptor with both operands MN-major (transpose bits 15, 16).
constexpr uint32_t kIdesc = idesc_bf16(kTM, kTN) | (1u << 15) | (1u << 16);

// TMA store of one box from shared memory (bulk-group completion) and its group waits.
__device__ __forceinline__ void tma_store_3d(const CUtensorMap* tm, uint32_t src, int c0, int c1, int c2) {
    asm volatile("cp.async.bulk.tensor.3d.global.shared::cta.bulk_group [%0, {%1, %2, %3}], [%4];" ::"l"(
                     (uint64_t)tm),
                 "r"(c0), "r"(c1), "r"(c2), "r"(src)
                 : "memory");
}
__device__ __forceinline__ void bulk_commit() { asm volatile("cp.async.bulk.commit_group;" ::: "memory"); }
__device__ __forceinline__ void bulk_wait_read1() { asm volatile("cp.async.bulk.wait_group.read 1;" ::: "memory"); }
__device__ __forceinline__ void bulk_wait_read0() { asm volatile("cp.async.bulk.wait_group.read 0;" ::: "memory"); }
__device__ __forceinline__ void bulk_wait_all() { asm volatile("cp.async.bulk.wait_group 0;" ::: "memory"); }

__global__ void __launch_bounds__(kThreads, 1)
materialize_tc_kernel(const __grid_constant__ CUtensorMap tmB, const __grid_constant__ CUtensorMap tmA,
                      const __grid_constant__ CUtensorMap tmG, const MParams p) {
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = (uint8_t*)(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
    uint8_t* outbuf = smem + (size_t)kStages * kStageBytes;  // 1024-byte aligned
    uint64_t* bars = (uint64_t*)(smem + (size_t)kStages * kStageBytes + kOutBytes);
    uint64_t* full = bars;                  // TMA bytes landed (count 1 + tx)
    uint64_t* empty = bars + kStages;       // MMAs done with the stage (count 1)
    uint64_t* tfull = bars + 2 * kStages;   // [2] accumulator ready
    uint64_t* tempty = tfull + 2;           // [2] accumulator drained (count 4)
    uint64_t* mma_done = tempty + 2;
    uint32_t* tmem_slot = (uint32_t*)(mma_done + 1);
    volatile int* abort = (volatile int*)(tmem_slot + 1);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    if (threadIdx.x == 0) {
        for (int s = 0; s < kStages; ++s) {
            mbar_init(smem_u32(&full[s]), 1);
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
    if (warp == 1) {
        tmem_alloc(smem_u32(tmem_slot), kTmemCols);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *tmem_slot;
    const int nk = p.nk;

    if (warp == 0) {
        if (lane == 0) {
            // ---------------- TMA producer: 2 + 4 boxes per stage
            uint32_t ring = 0, last_par[kStages];
            bool issued[kStages], ok = true;
            for (int s = 0; s < kStages; ++s) issued[s] = false;
            for (int64_t u = blockIdx.x; ok && u < p.n_units; u += gridDim.x) {
                const int e = (int)(u / (p.n_rb * p.n_cb));
                const int64_t rc = u % (p.n_rb * p.n_cb);
                const int r0 = (int)((rc / p.n_cb) * kTM), c0 = (int)((rc % p.n_cb) * kTN);
                for (int kc = 0; kc < nk; ++kc, ++ring) {
                    const int s = ring % kStages;
                    const uint32_t ph = (ring / kStages) & 1u;
                    if (!wait_bounded(smem_u32(&empty[s]), ph ^ 1u, abort, p.err)) {
                        ok = false;
                        break;
                    }
                    const uint32_t st = smem_u32(smem + (size_t)s * kStageBytes), bar = smem_u32(&full[s]);
                    mbar_arrive_tx(bar, kStageBytes);
#pragma unroll
                    for (int j = 0; j < kTM / 64; ++j) tma_load_3d(st + j * kBox, &tmB, r0 + 64 * j, kc * kTK, e, bar);
#pragma unroll
                    for (int j = 0; j < kTN / 64; ++j)
                        tma_load_3d(st + kABytes + j * kBox, &tmA, c0 + 64 * j, kc * kTK, e, bar);
                    issued[s] = true;
                    last_par[s] = ph;
                }
            }
            // copies still in flight when the MMA side stopped early land before the CTA exits
            for (int s = 0; s < kStages; ++s)
                if (issued[s]) {
                    const uint64_t t0 = global_ns();
                    while (!mbar_try_wait(smem_u32(&full[s]), last_par[s]))
                        if (global_ns() - t0 > kTimeoutNs) {
                            atomicOr(p.err, kErrTimeout);
                            break;
                        }
                }
        }
    } else if (warp == 1) {
        if (lane == 0) {
            // ---------------- MMA issuer
            uint32_t ring = 0, tile = 0;
            bool ok = true;
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
                    const uint32_t st = smem_u32(smem + (size_t)s * kStageBytes);
                    const uint64_t ad = sw128_mn_desc(st, kBox, 1024), bd = sw128_mn_desc(st + kABytes, kBox, 1024);
                    // 16 tokens per MMA = two 8-token groups = 2 KiB further into every box
#pragma unroll
                    for (int k = 0; k < kTK / 16; ++k)
                        mma_bf16(tmem + b * kTN, ad + (uint64_t)(k * 2048 >> 4), bd + (uint64_t)(k * 2048 >> 4),
                                 kIdesc, (kc > 0 || k > 0) ? 1u : 0u);
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
        // ---------------- epilogue: TMEM -> shared (swizzled 32 x 32 blocks) -> TMA store to G
        const int q = warp & 3;
        uint8_t* ob = outbuf + (size_t)(warp - 2) * 2 * kOutBox;
        uint32_t tile = 0, nblk = 0;
        bool prev_stored = false;  // lane 0: whether the previous block (the other buffer) went out
        for (int64_t u = blockIdx.x; u < p.n_units; u += gridDim.x, ++tile) {
            const uint32_t b = tile & 1u, use = tile >> 1;
            bool got = true;
            if (lane == 0) got = wait_bounded(smem_u32(&tfull[b]), use & 1u, abort, p.err);
            got = __shfl_sync(0xffffffffu, got, 0);
            if (epi_any(!got)) break;
            tc_fence_after();
            const int64_t e = u / (p.n_rb * p.n_cb), rc = u % (p.n_rb * p.n_cb);
            const int r0 = (int)((rc / p.n_cb) * kTM) + q * 32, c0 = (int)((rc % p.n_cb) * kTN);
            const uint32_t tb = tmem + ((uint32_t)(q * 32) << 16) + b * kTN;
#pragma unroll 1
            for (int c = 0; c < kTN; c += 32, ++nblk) {
                float v[32];
                tmem_ld16(tb + c, v);
                tmem_ld16(tb + c + 16, v + 16);
                uint8_t* blk = ob + (nblk & 1u) * kOutBox;
                // the store that last read this buffer (two blocks ago) has finished reading it:
                // at most one group, the other buffer's, may still be reading
                if (lane == 0) {
                    if (prev_stored)
                        bulk_wait_read1();
                    else
                        bulk_wait_read0();
                }
                __syncwarp();
                // row `lane`, 16-byte group j at chunk j ^ (row % 8): the 128-byte swizzle (conflict-free)
#pragma unroll
                for (int j = 0; j < 8; ++j)
                    *reinterpret_cast<float4*>(blk + lane * 128 + ((j ^ (lane & 7)) << 4)) =
                        make_float4(v[4 * j], v[4 * j + 1], v[4 * j + 2], v[4 * j + 3]);
                fence_proxy_async();
                __syncwarp();
                if (lane == 0) {
                    prev_stored = c0 + c < p.d_in && r0 < p.d_out;  // blocks wholly past the edge: nothing to store
                    if (prev_stored) {
                        tma_store_3d(&tmG, smem_u32(blk), c0 + c, r0, (int)e);
                        bulk_commit();
                    }
                }
            }
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(smem_u32(&tempty[b]));
        }
        if (lane == 0) bulk_wait_all();  // G written before the CTA exits
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 1) {
        tc_fence_after();
        tmem_dealloc(tmem, kTmemCols);
    }
}

// ---------------------------------------------------------------- host side
typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*, const cuuint64_t*,
                                  const cuuint64_t*, const cuuint32_t*, const cuuint32_t*, CUtensorMapInterleave,
                                  CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn encode_fn() {
    static EncodeTiledFn fn = nullptr;
    static std::once_flag once;
    std::call_once(once, [] {
        void* f = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &f, 12000, cudaEnableDefault, &q) ==
                cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = (EncodeTiledFn)f;
    });
    return fn;
}

// 3-D map over G[n][d_out][d_in] (fp32): box 32 columns x 32 rows x 1 example, 128-byte swizzle
// (stores are clipped at d_in and d_out).
bool make_map_out(CUtensorMap* tm, float* G, int64_t n, int64_t d_out, int64_t d_in) {
    EncodeTiledFn enc = encode_fn();
    if (!enc) return false;
    cuuint64_t dims[3] = {(cuuint64_t)d_in, (cuuint64_t)d_out, (cuuint64_t)n};
    cuuint64_t strides[2] = {(cuuint64_t)(d_in * 4), (cuuint64_t)(d_out * d_in * 4)};
    cuuint32_t box[3] = {32, 32, 1};
    cuuint32_t estr[3] = {1, 1, 1};
    return enc(tm, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 3, G, dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
               CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_NONE, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) ==
           CUDA_SUCCESS;
}

// 3-D map over X[n][T][d] (bf16): box 64 features x 64 tokens x 1 example, 128-byte swizzle, zero fill.
bool make_map(CUtensorMap* tm, const void* X, int64_t n, int64_t T, int64_t d) {
    EncodeTiledFn enc = encode_fn();
    if (!enc) return false;
    cuuint64_t dims[3] = {(cuuint64_t)d, (cuuint64_t)T, (cuuint64_t)n};
    cuuint64_t strides[2] = {(cuuint64_t)(d * 2), (cuuint64_t)(T * d * 2)};
    cuuint32_t box[3] = {64, (cuuint32_t)kTK, 1};
    cuuint32_t estr[3] = {1, 1, 1};
    return enc(tm, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(X), dims, strides, box, estr,
               CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
               CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
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
    // tensor maps: 16-byte row strides (d % 8), 32-bit token coordinates, example strides below 2^40 bytes
    const int64_t d_max = L.d_in > L.d_out ? L.d_in : L.d_out;
    return sm103 && encode_fn() && dt == TDA_BF16 && L.T >= 1 && L.T < ((int64_t)1 << 31) && L.d_in % 8 == 0 &&
           L.d_out % 8 == 0 && L.T * d_max * 2 < ((int64_t)1 << 40) && L.d_out * L.d_in * 4 < ((int64_t)1 << 40) &&
           L.d_in < ((int64_t)1 << 31) && L.d_out < ((int64_t)1 << 31) && ((uintptr_t)A & 15) == 0 &&
           ((uintptr_t)B & 15) == 0 && ((uintptr_t)G & 15) == 0;
}

// G[i][r][c] (i < n) of examples e0 .. e0+n-1 of bf16 factors A, B.
cudaError_t launch_materialize_tc(const tda_layer_desc& L, const void* A, const void* B, int64_t e0, int64_t n,
                                  float* G, unsigned int* err, cudaStream_t s) {
    if (n == 0) return cudaSuccess;
    // tensor-map coordinates are 32-bit: chunk the examples
    const int64_t max_n = ((int64_t)1 << 31) - 1;
    if (n > max_n) {
        for (int64_t i0 = 0; i0 < n; i0 += max_n) {
            const int64_t c = n - i0 < max_n ? n - i0 : max_n;
            cudaError_t e = launch_materialize_tc(L, A, B, e0 + i0, c, G + i0 * L.d_out * L.d_in, err, s);
            if (e != cudaSuccess) return e;
        }
        return cudaSuccess;
    }
    CUtensorMap mA, mB, mG;
    if (!make_map(&mA, (const __nv_bfloat16*)A + e0 * L.T * L.d_in, n, L.T, L.d_in) ||
        !make_map(&mB, (const __nv_bfloat16*)B + e0 * L.T * L.d_out, n, L.T, L.d_out) ||
        !make_map_out(&mG, G, n, L.d_out, L.d_in))
        return cudaErrorInvalidValue;
    MParams p;
    p.G = G;
    p.n = n;
    p.d_in = L.d_in;
    p.d_out = L.d_out;
    p.n_rb = (L.d_out + kTM - 1) / kTM;
    p.n_cb = (L.d_in + kTN - 1) / kTN;
    p.n_units = n * p.n_rb * p.n_cb;
    p.nk = (int)((L.T + kTK - 1) / kTK);
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
    materialize_tc_kernel<<<(unsigned)grid, kThreads, kSmem, s>>>(mB, mA, mG, p);
    return cudaGetLastError();
}

}  // namespace tda
