// k_gram_tc.cu -- route (c), the factored Gram identity (Eq. 4), on the
// tcgen05 tensor cores of sm_103a for bf16 factors:
//
//   <DW_q, DW_i>_F = sum_{t,s} (A_q A_i^T)[t][s] * (B_q B_i^T)[t][s].
//
// Both token Grams are dense contractions over the feature dimension, K-major
// in memory (a token's activations are contiguous), so they map directly onto
// tcgen05.mma: a 128-row tile of query tokens (M) against a 256-row tile of
// train tokens (N), K = d_in for X = A_q A_i^T and then K = d_out for
// Y = B_q B_i^T, both accumulators side by side in TMEM (2 x 256 columns). The
// epilogue reads each token row of X and Y, forms sum_s X[t][s] Y[t][s] over the
// columns of each train example and reduces over the rows of each query.
//
// Token tiles: for T <= 128 (a power of two) a query tile packs 128 / T query
// examples and a train tile 256 / T train examples, so one tile pair yields a
// whole block of S; for T >= 256 a (query, train) pair is a loop over its
// (T/128) x (T/256) tile pairs, summed in a register.
//
// Warp roles (256 threads, one persistent CTA per SM): warp 0 TMA producer,
// warp 1 TMEM allocator and MMA issuer (lane 0), warps 4-7 epilogue. Waits are
// bounded (about 1 s) and set kErrTimeout on expiry, as in the projection
// kernel.
#include <cuda.h>
#include <cuda_bf16.h>

#include <mutex>

#include "tda_internal.cuh"

namespace tda {
namespace {

constexpr int kThreads = 256;
constexpr int kTM = 128;                                 // query token rows per tile (MMA M)
constexpr int kTN = 256;                                 // train token rows per tile (MMA N)
constexpr int kChunkK = 64;                              // K elements per stage
constexpr uint32_t kABytes = kTM * kChunkK * 2;          // 16 KiB
constexpr uint32_t kBBytes = kTN * kChunkK * 2;          // 32 KiB
constexpr uint32_t kStageBytes = kABytes + kBBytes;
constexpr int kStages = 4;
constexpr uint32_t kTmemCols = 512;                      // X: 0..255, Y: 256..511
constexpr size_t kSmem = 1024 + (size_t)kStages * kStageBytes + 8 * 16 + 8 * (2 * kStages + 3) + 64;
static_assert(kSmem <= 232448, "shared memory per CTA");

struct GParams {
    int64_t n_q, n_t, T, ld_S;
    int nk_in, nk_out;
    int64_t n_units;      // tile pairs (T <= 128) or example pairs (T >= 256)
    int64_t n_qtiles;     // packed query tiles (T <= 128)
    int tiles_q, tiles_t; // token tiles per query / train example (T >= 256)
    float alpha, beta;
    float* S;
    unsigned int* err;
};

#include "tc_ptx.cuh"

__device__ __forceinline__ void emit(const GParams& p, int64_t q, int64_t i, float v) {
    float* dst = p.S + q * p.ld_S + i;
    *dst = p.beta == 0.f ? p.alpha * v : p.beta * (*dst) + p.alpha * v;
}

// sum over the rows of each query: lanes xor 1 .. R/2 (R <= 32) or the whole
// warp (R > 32); result valid in the first lane of each row group
__device__ __forceinline__ float row_reduce(float v, int R) {
    const int w = R < 32 ? R : 32;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1)
        if (o < w) v += __shfl_xor_sync(0xffffffffu, v, o);
    return v;
}

__global__ void __launch_bounds__(kThreads, 1)
gram_tc_kernel(const __grid_constant__ CUtensorMap tmAq, const __grid_constant__ CUtensorMap tmAt,
               const __grid_constant__ CUtensorMap tmBq, const __grid_constant__ CUtensorMap tmBt,
               const GParams p) {
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = (uint8_t*)(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
    float* red = (float*)(smem + (size_t)kStages * kStageBytes);   // [4 warps][4] cross-warp sums
    uint64_t* bars = (uint64_t*)(red + 16);
    uint64_t* full = bars;                 // stage landed (count 1 + tx)
    uint64_t* empty = bars + kStages;      // MMAs done with the stage
    uint64_t* tfull = bars + 2 * kStages;  // X, Y of a tile pair complete
    uint64_t* tempty = tfull + 1;          // epilogue drained TMEM (count 4)
    uint64_t* mma_done = tempty + 1;
    uint32_t* tmem_slot = (uint32_t*)(mma_done + 1);
    volatile int* abort = (volatile int*)(tmem_slot + 1);

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    if (threadIdx.x == 0) {
        for (int s = 0; s < kStages; ++s) {
            mbar_init(smem_u32(&full[s]), 1);
            mbar_init(smem_u32(&empty[s]), 1);
        }
        mbar_init(smem_u32(tfull), 1);
        mbar_init(smem_u32(tempty), 4);
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
    const bool packed = p.T <= kTM;
    const int nk_tot = p.nk_in + p.nk_out;
    const int tpp = packed ? 1 : p.tiles_q * p.tiles_t;  // tile pairs per unit

    if (warp == 0 && lane == 0) {
        // ---------------- TMA producer
        uint32_t ring = 0, last_par[kStages];
        bool issued[kStages], ok = true;
        for (int s = 0; s < kStages; ++s) issued[s] = false;
        for (int64_t u = blockIdx.x; ok && u < p.n_units; u += gridDim.x)
            for (int tp = 0; ok && tp < tpp; ++tp)
                for (int kc = 0; kc < nk_tot; ++kc, ++ring) {
                    const int s = ring % kStages;
                    const uint32_t ph = (ring / kStages) & 1u;
                    if (!wait_bounded(smem_u32(&empty[s]), ph ^ 1u, abort, p.err)) {
                        ok = false;
                        break;
                    }
                    const bool side_b = kc >= p.nk_in;
                    const int d0 = (side_b ? kc - p.nk_in : kc) * kChunkK;
                    int rq, eq, rt, et;
                    if (packed) {  // rows of the [n*T][d] views
                        rq = (int)((u % p.n_qtiles) * kTM);
                        rt = (int)((u / p.n_qtiles) * kTN);
                        eq = et = 0;
                    } else {       // token tiles of one query and one train example
                        eq = (int)(u % p.n_q);
                        et = (int)(u / p.n_q);
                        rq = (tp / p.tiles_t) * kTM;
                        rt = (tp % p.tiles_t) * kTN;
                    }
                    uint8_t* st = smem + (size_t)s * kStageBytes;
                    mbar_arrive_tx(smem_u32(&full[s]), kStageBytes);
                    tma_load_3d(smem_u32(st), side_b ? &tmBq : &tmAq, d0, rq, eq, smem_u32(&full[s]));
                    tma_load_3d(smem_u32(st + kABytes), side_b ? &tmBt : &tmAt, d0, rt, et, smem_u32(&full[s]));
                    issued[s] = true;
                    last_par[s] = ph;
                }
        for (int s = 0; s < kStages; ++s)
            if (issued[s]) {
                const uint64_t t0 = global_ns();
                while (!mbar_try_wait(smem_u32(&full[s]), last_par[s]))
                    if (global_ns() - t0 > kTimeoutNs) {
                        atomicOr(p.err, kErrTimeout);
                        break;
                    }
            }
    } else if (warp == 1 && lane == 0) {
        // ---------------- MMA issuer
        uint32_t ring = 0, pair = 0;
        bool ok = true;
        const uint32_t idesc = idesc_bf16(kTM, kTN);
        for (int64_t u = blockIdx.x; ok && u < p.n_units; u += gridDim.x)
            for (int tp = 0; ok && tp < tpp; ++tp, ++pair) {
                if (!wait_bounded(smem_u32(tempty), (pair & 1u) ^ 1u, abort, p.err)) {
                    ok = false;
                    break;
                }
                tc_fence_after();
                for (int kc = 0; kc < nk_tot; ++kc, ++ring) {
                    const int s = ring % kStages;
                    const uint32_t ph = (ring / kStages) & 1u;
                    if (!wait_bounded(smem_u32(&full[s]), ph, abort, p.err)) {
                        ok = false;
                        break;
                    }
                    tc_fence_after();
                    const bool side_b = kc >= p.nk_in;
                    const int kk = side_b ? kc - p.nk_in : kc;
                    uint8_t* st = smem + (size_t)s * kStageBytes;
                    const uint64_t ad = sw128_desc(smem_u32(st)), bd = sw128_desc(smem_u32(st + kABytes));
                    const uint32_t d_tmem = tmem + (side_b ? (uint32_t)kTN : 0u);
#pragma unroll
                    for (int k = 0; k < kChunkK / 16; ++k)
                        mma_bf16(d_tmem, ad + 2 * k, bd + 2 * k, idesc, (kk > 0 || k > 0) ? 1u : 0u);
                    mma_commit(smem_u32(&empty[s]));
                }
                if (!ok) break;
                mma_commit(smem_u32(tfull));
            }
        mma_commit(smem_u32(mma_done));
        const uint64_t t0 = global_ns();
        while (!mbar_try_wait(smem_u32(mma_done), 0))
            if (global_ns() - t0 > kTimeoutNs) {
                atomicOr(p.err, kErrTimeout);
                break;
            }
    } else if (warp >= 4) {
        // ---------------- epilogue
        const int q4 = warp & 3, row = q4 * 32 + lane;
        const int R = packed ? (int)p.T : kTM;   // rows per query in a tile
        const int Cg = packed ? (int)p.T : kTN;  // columns per train example in a tile
        const uint32_t lane_base = tmem + ((uint32_t)(q4 * 32) << 16);
        uint32_t pair = 0;
        bool stop = false;
        for (int64_t u = blockIdx.x; !stop && u < p.n_units; u += gridDim.x) {
            float pair_acc = 0.f;  // T >= 256: running sum of this (query, train) pair
            for (int tp = 0; tp < tpp; ++tp, ++pair) {
                bool got = true;
                if (lane == 0) got = wait_bounded(smem_u32(tfull), pair & 1u, abort, p.err);
                got = __shfl_sync(0xffffffffu, got, 0);
                if (epi_any(!got)) {
                    stop = true;
                    break;
                }
                tc_fence_after();
                float part = 0.f;
                int g = 0;  // column group (train example within the tile)
                for (int c0 = 0; c0 < kTN; c0 += 16) {
                    float x[16], y[16];
                    tmem_ld16(lane_base + c0, x);
                    tmem_ld16(lane_base + kTN + c0, y);
#pragma unroll
                    for (int c = 0; c < 16; ++c) {
                        part = fmaf(x[c], y[c], part);
                        if (((c0 + c + 1) % Cg) == 0) {
                            // one train example's columns done for this row
                            if (packed) {
                                float v = row_reduce(part, R);
                                const int64_t qi = (u % p.n_qtiles) * (kTM / R) + row / R;
                                const int64_t ti = (u / p.n_qtiles) * (kTN / Cg) + g;
                                if (R <= 32) {
                                    if ((lane & (R - 1)) == 0 && qi < p.n_q && ti < p.n_t) emit(p, qi, ti, v);
                                } else {
                                    // rows of one query span R / 32 warps
                                    if (lane == 0) red[q4 * 4 + (g & 3)] = v;
                                    epi_sync();
                                    if (lane == 0 && (q4 % (R / 32)) == 0) {
                                        float s = 0.f;
                                        for (int w = 0; w < R / 32; ++w) s += red[(q4 + w) * 4 + (g & 3)];
                                        if (qi < p.n_q && ti < p.n_t) emit(p, qi, ti, s);
                                    }
                                    epi_sync();
                                }
                            }
                            ++g;
                            if (packed) part = 0.f;
                        }
                    }
                }
                tc_fence_before();
                __syncwarp();
                if (lane == 0) mbar_arrive(smem_u32(tempty));
                if (!packed) {
                    // the whole tile belongs to one (query, train) pair
                    float v = row_reduce(part, 32);
                    if (lane == 0) red[q4] = v;
                    epi_sync();
                    if (threadIdx.x == 128) pair_acc += red[0] + red[1] + red[2] + red[3];
                    epi_sync();
                }
            }
            if (!stop && !packed && threadIdx.x == 128) emit(p, u % p.n_q, u / p.n_q, pair_acc);
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

// 3-D map over X[n][rows][d] (bf16), box 64 (d) x box_rows x 1, 128B swizzle, zero fill.
bool make_map(CUtensorMap* tm, const void* X, int64_t n, int64_t rows, int64_t d, int box_rows) {
    EncodeTiledFn enc = encode_fn();
    if (!enc) return false;
    cuuint64_t dims[3] = {(cuuint64_t)d, (cuuint64_t)rows, (cuuint64_t)n};
    cuuint64_t strides[2] = {(cuuint64_t)(d * 2), (cuuint64_t)(rows * d * 2)};
    cuuint32_t box[3] = {kChunkK, (cuuint32_t)box_rows, 1};
    cuuint32_t estr[3] = {1, 1, 1};
    return enc(tm, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(X), dims, strides, box, estr,
               CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
               CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

bool is_pow2(int64_t v) { return v > 0 && (v & (v - 1)) == 0; }

}  // namespace

bool gram_tc_supported(const tda_layer_desc& L, tda_dtype dt, const void* Aq, const void* Bq, const void* At,
                       const void* Bt) {
    static int sm103 = -1;
    if (sm103 < 0) {
        int dev = 0, major = 0, minor = 0;
        cudaGetDevice(&dev);
        cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev);
        cudaDeviceGetAttribute(&minor, cudaDevAttrComputeCapabilityMinor, dev);
        sm103 = (major == 10 && minor == 3) ? 1 : 0;
    }
    if (!sm103 || !encode_fn() || dt != TDA_BF16) return false;
    if (!is_pow2(L.T) || L.T > (1 << 20) || L.d_in % 8 || L.d_out % 8) return false;
    for (const void* x : {Aq, Bq, At, Bt})
        if ((uintptr_t)x & 15) return false;
    return true;
}

// S[q][i] = beta * S[q][i] + alpha * <DW_q, DW_i>_F for bf16 factors.
cudaError_t launch_gram_tc(const tda_layer_desc& L, const void* Aq, const void* Bq, int64_t n_q, const void* At,
                           const void* Bt, int64_t n_t, float* S, int64_t ld_S, float beta, float alpha,
                           unsigned int* err, cudaStream_t s) {
    if (n_q == 0 || n_t == 0) return cudaSuccess;
    const int64_t T = L.T;
    const bool packed = T <= kTM;
    const int64_t d_max = L.d_in > L.d_out ? L.d_in : L.d_out;
    if (packed) {
        // 32-bit TMA row coordinates and strides below 2^40 bytes: split the train side
        int64_t max_t = ((int64_t)1 << 30) / T;
        const int64_t by_stride = (((int64_t)1 << 40) - 1) / (T * d_max * 2);
        if (by_stride < max_t) max_t = by_stride;
        max_t = max_t / (kTN / T) * (kTN / T);
        if (n_q * T >= ((int64_t)1 << 30) || n_q > by_stride || max_t < 1) return cudaErrorInvalidValue;
        if (n_t > max_t) {
            for (int64_t i0 = 0; i0 < n_t; i0 += max_t) {
                const int64_t n = n_t - i0 < max_t ? n_t - i0 : max_t;
                cudaError_t e = launch_gram_tc(L, Aq, Bq, n_q, (const char*)At + i0 * T * L.d_in * 2,
                                               (const char*)Bt + i0 * T * L.d_out * 2, n, S + i0, ld_S, beta,
                                               alpha, err, s);
                if (e != cudaSuccess) return e;
            }
            return cudaSuccess;
        }
    }
    CUtensorMap mAq, mAt, mBq, mBt;
    bool ok;
    if (packed)
        ok = make_map(&mAq, Aq, 1, n_q * T, L.d_in, kTM) && make_map(&mAt, At, 1, n_t * T, L.d_in, kTN) &&
             make_map(&mBq, Bq, 1, n_q * T, L.d_out, kTM) && make_map(&mBt, Bt, 1, n_t * T, L.d_out, kTN);
    else
        ok = make_map(&mAq, Aq, n_q, T, L.d_in, kTM) && make_map(&mAt, At, n_t, T, L.d_in, kTN) &&
             make_map(&mBq, Bq, n_q, T, L.d_out, kTM) && make_map(&mBt, Bt, n_t, T, L.d_out, kTN);
    if (!ok) return cudaErrorInvalidValue;
    GParams p;
    p.n_q = n_q;
    p.n_t = n_t;
    p.T = T;
    p.ld_S = ld_S;
    p.nk_in = (int)((L.d_in + kChunkK - 1) / kChunkK);
    p.nk_out = (int)((L.d_out + kChunkK - 1) / kChunkK);
    p.tiles_q = packed ? 1 : (int)(T / kTM);
    p.tiles_t = packed ? 1 : (int)(T / kTN);
    if (packed) {
        p.n_qtiles = (n_q * T + kTM - 1) / kTM;
        p.n_units = p.n_qtiles * ((n_t * T + kTN - 1) / kTN);
    } else {
        p.n_qtiles = 0;
        p.n_units = n_q * n_t;
    }
    p.alpha = alpha;
    p.beta = beta;
    p.S = S;
    p.err = err;
    static int sms = 0;
    if (!sms) {
        int dev = 0;
        cudaGetDevice(&dev);
        cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
        if (sms <= 0) sms = 1;
    }
    cudaError_t e = cudaFuncSetAttribute(gram_tc_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kSmem);
    if (e != cudaSuccess) return e;
    const int64_t grid = p.n_units < sms ? p.n_units : sms;
    note_launches(1);
    gram_tc_kernel<<<(unsigned)grid, kThreads, kSmem, s>>>(mAq, mAt, mBq, mBt, p);
    return cudaGetLastError();
}

}  // namespace tda
