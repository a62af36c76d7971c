// k_tokens_tc.cu -- token-level scores on the tcgen05 tensor cores (3xTF32):
//   out[q][t] = beta * out[q][t] + scale * g~_t^T R_q a~_t
// for k_in = 32 and k_out in {16, 32, 64} (the token-level decomposition of
// the score: summed over t it gives <Phi_i, R_q>).
//
// As a contraction: X[t][(q, r)] = sum_c a~_t[c] R_q[r][c] is a GEMM with
// M = 128 tokens, N = 256 rows (q, r) of the stacked query matrices, K = k_in;
// the epilogue weights X by g~_t[r] and sums over r, one output per (t, q).
// fp32 accuracy from TF32 tensor cores as in the score GEMM: x = hi + lo,
// products hi*hi + hi*lo + lo*hi.
//
// Shared memory: two token-tile buffers (a~ hi and lo, 16 KiB each) and a ring
// of two query stages (R hi and lo, 32 KiB each, split once per call into the
// workspace). All tiles are K-major with 128-byte rows (32 fp32) and the
// 128-byte swizzle that TMA writes.
//
// Warp roles (256 threads, so that no SM sub-partition holds more than two
// warps and every thread may use up to 255 registers): warps 0 and 3 split the
// token tile in place (hi stays, lo goes to its own tile); warp 1 allocates
// TMEM, its lane 0 issues the MMAs into two 256-column fp32 accumulators; lane
// 0 of warp 2 issues the TMA copies; warps 4-7 are the epilogue (TMEM lane
// quadrant warp % 4). Waits are bounded (about 1 s) and set kErrTimeout on
// expiry.
#include <cuda.h>

#include <mutex>

#include "tda_internal.cuh"

namespace tda {
namespace {

#include "tc_ptx.cuh"

constexpr int kThreads = 256;
constexpr int kTM = 128;                          // tokens per tile
constexpr int kTN = 256;                          // (query, r) rows per stage
constexpr int kKA = 32;                           // k_in: one 128-byte operand row
constexpr uint32_t kATile = kTM * kKA * 4;        // 16 KiB
constexpr uint32_t kBTile = kTN * kKA * 4;        // 32 KiB
constexpr uint32_t kABuf = 2 * kATile;            // hi + lo
constexpr uint32_t kBBuf = 2 * kBTile;
constexpr uint32_t kTmemCols = 512;
constexpr size_t kSmem = 1024 + 2 * (size_t)kABuf + 2 * (size_t)kBBuf + 8 * 17 + 16;
static_assert(kSmem <= 232448, "shared memory per CTA");

struct TParams {
    const float* Yb;   // g~ rows [NT][k_out]
    float* out;
    int64_t NT;        // tokens of this call
    int64_t tok0;      // global token index of token 0 (first example of the call times T)
    int64_t n_q, ld_q;
    int n_tt, n_nt;    // token tiles, query stages
    float scale, beta;
    unsigned int* err;
};

__host__ __device__ constexpr uint32_t idesc_tf32(int M, int N) {
    return (1u << 4) | (2u << 7) | (2u << 10) | ((uint32_t)(N >> 3) << 17) | ((uint32_t)(M >> 4) << 24);
}
__device__ __forceinline__ void mma_tf32(uint32_t d_tmem, uint64_t adesc, uint64_t bdesc, uint32_t idesc,
                                         uint32_t accumulate) {
    asm volatile(
        "{\n .reg .pred p;\n setp.ne.b32 p, %4, 0;\n tcgen05.mma.cta_group::1.kind::tf32 [%0], %1, %2, %3, p;\n}" ::"r"(
            d_tmem),
        "l"(adesc), "l"(bdesc), "r"(idesc), "r"(accumulate)
        : "memory");
}
__device__ __forceinline__ void split_tf32(float x, float& hi, float& lo) {
    hi = __uint_as_float(__float_as_uint(x) & 0xFFFFE000u);
    lo = x - hi;
}
__device__ __forceinline__ void tma_load_2d(uint32_t dst, const CUtensorMap* tm, int c0, int c1, uint32_t bar) {
    asm volatile(
        "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3}], [%4];" ::"r"(
            dst),
        "l"((uint64_t)tm), "r"(c0), "r"(c1), "r"(bar)
        : "memory");
}
// bounded wait on the phase `parity` of `bar` without an abort flag (teardown drains)
__device__ __forceinline__ void drain_wait(uint32_t bar, uint32_t parity, unsigned int* err) {
    const uint64_t t0 = global_ns();
    while (!mbar_try_wait(bar, parity))
        if (global_ns() - t0 > kTimeoutNs) {
            atomicOr(err, kErrTimeout);
            break;
        }
}

// hi/lo halves of R: row (q, r) of Rs = R[q * ld_R + r * 32 + c]
__global__ void split_r_kernel(const float* __restrict__ R, int64_t n_q, int64_t ld_R, int kg, float* __restrict__ Rhi,
                               float* __restrict__ Rlo) {
    const int64_t per = (int64_t)kg * kKA, total = n_q * per;
    for (int64_t e = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; e < total; e += (int64_t)gridDim.x * blockDim.x) {
        const int64_t q = e / per, rc = e - q * per;
        float h, l;
        split_tf32(R[q * ld_R + rc], h, l);
        Rhi[e] = h;
        Rlo[e] = l;
    }
}

template <int KG>
__global__ void __launch_bounds__(kThreads, 1)
token_tc_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmRh,
                const __grid_constant__ CUtensorMap tmRl, const TParams p) {
    constexpr int G = kTN / KG;  // queries per stage
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = (uint8_t*)(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
    uint8_t* abuf = smem;                  // [2] a~ hi | lo
    uint8_t* bbuf = smem + 2 * kABuf;      // [2] R hi | lo
    uint64_t* bars = (uint64_t*)(bbuf + 2 * kBBuf);
    uint64_t* a_raw = bars;        // [2] TMA landed (1 + tx)
    uint64_t* a_full = bars + 2;   // [2] split done (2 warps)
    uint64_t* a_empty = bars + 4;  // [2] MMAs done with the token tile (commit)
    uint64_t* b_full = bars + 6;   // [2] (1 + tx)
    uint64_t* b_empty = bars + 8;  // [2] (commit)
    uint64_t* tfull = bars + 10;   // [2] accumulator ready (commit)
    uint64_t* tempty = bars + 12;  // [2] accumulator drained (4)
    uint64_t* mma_done = bars + 14;
    uint32_t* tmem_slot = (uint32_t*)(bars + 17);
    volatile int* abort = (volatile int*)(tmem_slot + 1);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    if (threadIdx.x == 0) {
        for (int i = 0; i < 2; ++i) {
            mbar_init(smem_u32(&a_raw[i]), 1);
            mbar_init(smem_u32(&a_full[i]), 2);
            mbar_init(smem_u32(&a_empty[i]), 1);
            mbar_init(smem_u32(&b_full[i]), 1);
            mbar_init(smem_u32(&b_empty[i]), 1);
            mbar_init(smem_u32(&tfull[i]), 1);
            mbar_init(smem_u32(&tempty[i]), 4);
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

    if (warp == 0 || warp == 3) {
        // ---------------- split warps: a~ tile raw (TMA) -> hi in place + lo
        const int pt = (warp == 0 ? 0 : 32) + lane;
        uint32_t it = 0;
        for (int u = blockIdx.x; u < p.n_tt; u += gridDim.x, ++it) {
            const uint32_t ab = it & 1u, ph = (it >> 1) & 1u;
            bool got = true;
            if (lane == 0) got = wait_bounded(smem_u32(&a_raw[ab]), ph, abort, p.err);
            got = __shfl_sync(0xffffffffu, got, 0);
            if (!got) break;
            uint8_t* hi = abuf + ab * kABuf;
            uint8_t* lo = hi + kATile;
#pragma unroll 4
            for (uint32_t off = (uint32_t)pt * 16u; off < kATile; off += 64u * 16u) {
                const float4 v = *reinterpret_cast<const float4*>(hi + off);
                float4 h, l;
                split_tf32(v.x, h.x, l.x);
                split_tf32(v.y, h.y, l.y);
                split_tf32(v.z, h.z, l.z);
                split_tf32(v.w, h.w, l.w);
                *reinterpret_cast<float4*>(hi + off) = h;
                *reinterpret_cast<float4*>(lo + off) = l;
            }
            fence_proxy_async();
            __syncwarp();
            if (lane == 0) mbar_arrive(smem_u32(&a_full[ab]));
        }
    } else if (warp == 1) {
        if (lane == 0) {
            // ---------------- MMA issuer
            constexpr uint32_t idesc = idesc_tf32(kTM, kTN);
            uint32_t it = 0, rb = 0, tt = 0;
            bool ok = true;
            for (int u = blockIdx.x; ok && u < p.n_tt; u += gridDim.x, ++it) {
                const uint32_t ab = it & 1u;
                if (!wait_bounded(smem_u32(&a_full[ab]), (it >> 1) & 1u, abort, p.err)) break;
                tc_fence_after();
                const uint32_t ahs = smem_u32(abuf + ab * kABuf);
                const uint64_t ahi = sw128_desc(ahs), alo = sw128_desc(ahs + kATile);
                for (int j = 0; j < p.n_nt; ++j, ++rb, ++tt) {
                    const uint32_t s = rb & 1u, b = tt & 1u;
                    if (!wait_bounded(smem_u32(&tempty[b]), ((tt >> 1) & 1u) ^ 1u, abort, p.err) ||
                        !wait_bounded(smem_u32(&b_full[s]), (rb >> 1) & 1u, abort, p.err)) {
                        ok = false;
                        break;
                    }
                    tc_fence_after();
                    const uint32_t bhs = smem_u32(bbuf + s * kBBuf);
                    const uint64_t bhi = sw128_desc(bhs), blo = sw128_desc(bhs + kBTile);
                    const uint32_t d = tmem + b * kTN;
#pragma unroll
                    for (int k = 0; k < kKA / 8; ++k) {  // K = 8 tf32 = 32 bytes per instruction
                        mma_tf32(d, ahi + 2 * k, bhi + 2 * k, idesc, k > 0 ? 1u : 0u);
                        mma_tf32(d, ahi + 2 * k, blo + 2 * k, idesc, 1u);
                        mma_tf32(d, alo + 2 * k, bhi + 2 * k, idesc, 1u);
                    }
                    mma_commit(smem_u32(&b_empty[s]));
                    mma_commit(smem_u32(&tfull[b]));
                }
                if (!ok) break;
                mma_commit(smem_u32(&a_empty[ab]));
            }
            mma_commit(smem_u32(mma_done));
            drain_wait(smem_u32(mma_done), 0, p.err);
        }
    } else if (warp == 2) {
        if (lane == 0) {
            // ---------------- TMA producer
            uint32_t it = 0, rb = 0;
            uint32_t a_par[2], b_par[2];
            bool a_iss[2] = {false, false}, b_iss[2] = {false, false}, ok = true;
            for (int u = blockIdx.x; ok && u < p.n_tt; u += gridDim.x, ++it) {
                const uint32_t ab = it & 1u, aph = (it >> 1) & 1u;
                if (!wait_bounded(smem_u32(&a_empty[ab]), aph ^ 1u, abort, p.err)) break;
                mbar_arrive_tx(smem_u32(&a_raw[ab]), kATile);
                tma_load_2d(smem_u32(abuf + ab * kABuf), &tmA, 0, u * kTM, smem_u32(&a_raw[ab]));
                a_iss[ab] = true;
                a_par[ab] = aph;
                for (int j = 0; j < p.n_nt; ++j, ++rb) {
                    const uint32_t s = rb & 1u, ph = (rb >> 1) & 1u;
                    if (!wait_bounded(smem_u32(&b_empty[s]), ph ^ 1u, abort, p.err)) {
                        ok = false;
                        break;
                    }
                    const uint32_t dst = smem_u32(bbuf + s * kBBuf), bar = smem_u32(&b_full[s]);
                    mbar_arrive_tx(bar, kBBuf);
                    tma_load_2d(dst, &tmRh, 0, j * kTN, bar);
                    tma_load_2d(dst + kBTile, &tmRl, 0, j * kTN, bar);
                    b_iss[s] = true;
                    b_par[s] = ph;
                }
            }
            // copies still in flight when the consumers stopped early land before the CTA exits
            for (int i = 0; i < 2; ++i) {
                if (a_iss[i]) drain_wait(smem_u32(&a_raw[i]), a_par[i], p.err);
                if (b_iss[i]) drain_wait(smem_u32(&b_full[i]), b_par[i], p.err);
            }
        }
    } else {
        // ---------------- epilogue: TMEM -> weighted sums over r -> out
        const int q4 = warp & 3, row = q4 * 32 + lane;
        uint32_t tt = 0;
        bool stop = false;
        for (int u = blockIdx.x; !stop && u < p.n_tt; u += gridDim.x) {
            const int64_t tok = (int64_t)u * kTM + row;
            const bool valid = tok < p.NT;
            float g[KG];
#pragma unroll
            for (int c = 0; c < KG; c += 4) {
                float4 v = make_float4(0.f, 0.f, 0.f, 0.f);
                if (valid) v = *reinterpret_cast<const float4*>(p.Yb + tok * KG + c);
                g[c] = v.x, g[c + 1] = v.y, g[c + 2] = v.z, g[c + 3] = v.w;
            }
            // beta != 0: the previous values of a stage's outputs are loaded one stage ahead,
            // so that their latency hides behind the wait for the accumulator
            const bool rmw = p.beta != 0.f;
            float old[G];
            auto prefetch = [&](int j) {
#pragma unroll
                for (int gq = 0; gq < G; ++gq) {
                    const int64_t q = (int64_t)j * G + gq;
                    old[gq] = (rmw && valid && q < p.n_q) ? p.out[q * p.ld_q + p.tok0 + tok] : 0.f;
                }
            };
            prefetch(0);
            for (int j = 0; j < p.n_nt; ++j, ++tt) {
                const uint32_t b = tt & 1u;
                bool got = true;
                if (lane == 0) got = wait_bounded(smem_u32(&tfull[b]), (tt >> 1) & 1u, abort, p.err);
                got = __shfl_sync(0xffffffffu, got, 0);
                if (epi_any(!got)) {
                    stop = true;
                    break;
                }
                tc_fence_after();
                const uint32_t tb = tmem + ((uint32_t)(q4 * 32) << 16) + b * kTN;
                float acc[G];
#pragma unroll
                for (int gq = 0; gq < G; ++gq) {
                    float s = 0.f;
#pragma unroll
                    for (int c = 0; c < KG; c += 16) {
                        float v[16];
                        tmem_ld16(tb + gq * KG + c, v);
#pragma unroll
                        for (int i = 0; i < 16; ++i) s = fmaf(g[c + i], v[i], s);
                    }
                    acc[gq] = rmw ? p.beta * old[gq] + p.scale * s : p.scale * s;
                }
                tc_fence_before();
                __syncwarp();
                if (lane == 0) mbar_arrive(smem_u32(&tempty[b]));
                if (valid) {
#pragma unroll
                    for (int gq = 0; gq < G; ++gq) {
                        const int64_t q = (int64_t)j * G + gq;
                        if (q < p.n_q) p.out[q * p.ld_q + p.tok0 + tok] = acc[gq];
                    }
                }
                if (j + 1 < p.n_nt) prefetch(j + 1);
            }
        }
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

// 2-D map over fp32 rows of 32 elements: box 32 x box_rows, 128-byte swizzle, zero fill past the last row.
bool make_rows_map(CUtensorMap* tm, const float* X, int64_t rows, int box_rows) {
    EncodeTiledFn enc = encode_fn();
    if (!enc) return false;
    cuuint64_t dims[2] = {(cuuint64_t)kKA, (cuuint64_t)rows};
    cuuint64_t strides[1] = {(cuuint64_t)(kKA * 4)};
    cuuint32_t box[2] = {(cuuint32_t)kKA, (cuuint32_t)box_rows};
    cuuint32_t estr[2] = {1, 1};
    return enc(tm, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 2, const_cast<float*>(X), dims, strides, box, estr,
               CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
               CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

bool is_sm103() {
    static int sm103 = -1;
    if (sm103 < 0) {
        int dev = 0, major = 0, minor = 0;
        cudaGetDevice(&dev);
        cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev);
        cudaDeviceGetAttribute(&minor, cudaDevAttrComputeCapabilityMinor, dev);
        sm103 = (major == 10 && minor == 3) ? 1 : 0;
    }
    return sm103 == 1;
}

}  // namespace

size_t token_tc_split_bytes(int ka, int kg, int64_t n_q) {
    return (2 * sizeof(float) * (size_t)n_q * (size_t)ka * (size_t)kg + 255) & ~(size_t)255;
}

bool token_tc_supported(int ka, int kg, int64_t n_q) {
    return is_sm103() && encode_fn() && ka == kKA && (kg == 16 || kg == 32 || kg == 64) && n_q >= 1 &&
           n_q * kg < ((int64_t)1 << 31) && device_error_word() != nullptr;
}

// Rs: token_tc_split_bytes(ka, kg, n_q) of device scratch for R's hi and lo halves.
cudaError_t launch_token_scores_tc(const float* Ya, const float* Yb, int64_t n, int64_t T, int ka, int kg,
                                   const float* R, int64_t n_q, int64_t ld_R, float scale, float* out, int64_t ld_q,
                                   int64_t i0, float beta, float* Rs, cudaStream_t s) {
    const int64_t NT = n * T;
    if (NT == 0 || n_q == 0) return cudaSuccess;
    if (NT >= ((int64_t)1 << 31) || ((uintptr_t)Ya & 15) || ((uintptr_t)Yb & 15) || ((uintptr_t)Rs & 15))
        return cudaErrorInvalidValue;
    float* Rhi = Rs;
    float* Rlo = Rs + n_q * kg * ka;
    CUtensorMap mA, mRh, mRl;
    if (!make_rows_map(&mA, Ya, NT, kTM) || !make_rows_map(&mRh, Rhi, n_q * kg, kTN) ||
        !make_rows_map(&mRl, Rlo, n_q * kg, kTN))
        return cudaErrorInvalidValue;
    note_launches(1);
    split_r_kernel<<<(unsigned)((n_q * kg * ka + 255) / 256 < 1024 ? (n_q * kg * ka + 255) / 256 : 1024), 256, 0, s>>>(
        R, n_q, ld_R, kg, Rhi, Rlo);
    TParams p;
    p.Yb = Yb;
    p.out = out;
    p.NT = NT;
    p.tok0 = i0 * T;
    p.n_q = n_q;
    p.ld_q = ld_q;
    p.n_tt = (int)((NT + kTM - 1) / kTM);
    p.n_nt = (int)((n_q * kg + kTN - 1) / kTN);
    p.scale = scale;
    p.beta = beta;
    p.err = device_error_word();
    static int sms = 0;
    if (!sms) {
        int dev = 0;
        cudaGetDevice(&dev);
        cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
        if (sms <= 0) sms = 1;
    }
    const unsigned grid = (unsigned)(p.n_tt < sms ? p.n_tt : sms);
    cudaError_t e;
    note_launches(1);
    if (kg == 16) {
        if ((e = cudaFuncSetAttribute(token_tc_kernel<16>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kSmem)))
            return e;
        token_tc_kernel<16><<<grid, kThreads, kSmem, s>>>(mA, mRh, mRl, p);
    } else if (kg == 32) {
        if ((e = cudaFuncSetAttribute(token_tc_kernel<32>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kSmem)))
            return e;
        token_tc_kernel<32><<<grid, kThreads, kSmem, s>>>(mA, mRh, mRl, p);
    } else {
        if ((e = cudaFuncSetAttribute(token_tc_kernel<64>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kSmem)))
            return e;
        token_tc_kernel<64><<<grid, kThreads, kSmem, s>>>(mA, mRh, mRl, p);
    }
    return cudaGetLastError();
}

}  // namespace tda
