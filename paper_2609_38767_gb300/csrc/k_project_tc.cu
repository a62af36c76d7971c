// k_project_tc.cu -- factored projection (Eq. 2) on the 5th-generation tensor
// cores of sm_103a: tcgen05.mma with TMEM accumulators, operands staged in
// shared memory by TMA (factors) and by a generator warp (signs).
//
// For every example n and every 128-token tile of it:
//   At = A_tile S_in   (128 x k_in,  K = d_in)    tcgen05, accumulators in TMEM
//   Bt = B_tile S_out  (128 x k_out, K = d_out)   tcgen05, accumulators in TMEM
//   Phi_n += Bt^T At   (k_out x k_in, over the 128 tokens) on CUDA cores, fp32
// and finally Phi_n *= 1/sqrt(k_in k_out). The signs S (App. A.2) come from the
// counter hash: one 64-bit word gives the 64 signs of one column over one
// 64-row K chunk, which is one 128-byte row of the K-major, 128B-swizzled
// operand tile, so the projection matrices never touch global memory.
//
// The kernel streams every factor byte once from HBM; at k <= 64 its
// arithmetic intensity (~k flop/B) is far below the tensor-core ridge, so it
// is HBM-bound and the pipeline is sized for bytes in flight.
//
// Warp roles (256 threads, one persistent CTA per SM):
//   warp 0  TMA producer: 128x64 bf16 factor tiles into the stage ring
//   warp 1  TMEM allocator; lane 0 issues the MMAs
//   warps 2-3  sign generators: k x 64 bf16 +-1 tiles into the stage ring,
//           each warp one half of every 128-byte row (one warp alone falls
//           behind the HBM stream)
//   warps 4-7  epilogue: TMEM -> registers -> shared -> token contraction
// Accumulators are double-buffered in TMEM, so the epilogue of one tile
// overlaps the MMAs of the next. Every wait is bounded (about 1 s); on expiry
// the kernel records kErrTimeout in the device error word, drains its copies,
// frees its TMEM and returns.
#include <cuda.h>
#include <cuda_bf16.h>

#include <mutex>

#include "tda_internal.cuh"

namespace tda {
namespace {

constexpr int kThreads = 256;
constexpr int kTileM = 128;            // tokens per tile (MMA M)
constexpr int kChunkK = 64;            // K elements per stage (128 bytes of bf16)
constexpr uint32_t kTileBytes = kTileM * kChunkK * 2;  // 16 KiB per factor tile

template <int K>
struct Cfg {
    static constexpr int kStages = K <= 32 ? 8 : 6;
    static constexpr uint32_t kSignBytes = K * 128;  // K rows x 128 bytes
    static constexpr int kStageLd = K + 4;           // padded fp32 staging row
    static constexpr int kAccCols = 2 * K;           // At | Bt in one accumulator buffer
    static constexpr uint32_t kTmemCols = 2 * kAccCols < 32 ? 32 : 2 * kAccCols;
    static constexpr size_t kSmemA = (size_t)kStages * kTileBytes;
    static constexpr size_t kSmemS = (size_t)kStages * kSignBytes;
    static constexpr size_t kSmemStage = 2ull * kTileM * kStageLd * 4;
    static constexpr size_t kSmemBars = 8 * (3 * kStages + 7) + 16;
    static constexpr size_t kSmem = 1024 + kSmemA + kSmemS + kSmemStage + kSmemBars;
    // contraction blocking: 16 row groups x 8 column groups of threads
    static constexpr int RB = K / 16 > 0 ? K / 16 : 1;
    static constexpr int CB = K / 8;
};

struct Params {
    int64_t N, T, d_in, d_out, ld_phi;
    uint64_t key_in, key_out;
    float scale;
    float* phi;
    unsigned int* err;
    int n_ttiles, nk_in, nk_out;
    int cs;  // CTAs per cluster sharing one example's token tiles (1, 2 or 4)
};

#include "tc_ptx.cuh"

// Half `half` (16-byte chunks 4*half .. 4*half+3) of row n of a K-major
// 128B-swizzled sign tile: signs of column n over the K chunk, as bf16 +1
// (0x3F80) or -1 (0xBF80). Two generator warps each write one half.
__device__ __forceinline__ void write_sign_half(uint8_t* tile, int n, uint64_t w, int half) {
    uint8_t* row = tile + (n >> 3) * 1024 + (n & 7) * 128;
#pragma unroll
    for (int cc = 0; cc < 4; ++cc) {
        const int c = cc + 4 * half;
        const uint32_t bits = (uint32_t)(w >> (8 * c)) & 0xFFu;
        uint32_t q[4];
#pragma unroll
        for (int p = 0; p < 4; ++p) {
            const uint32_t lo = 0x3F80u | (((bits >> (2 * p)) & 1u) << 15);
            const uint32_t hi = 0x3F80u | (((bits >> (2 * p + 1)) & 1u) << 15);
            q[p] = lo | (hi << 16);
        }
        *reinterpret_cast<uint4*>(row + ((c ^ (n & 7)) << 4)) = make_uint4(q[0], q[1], q[2], q[3]);
    }
}

template <int K>
__global__ void __launch_bounds__(kThreads, 1)
project_tc_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
                  const Params p) {
    using C = Cfg<K>;
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = (uint8_t*)(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
    uint8_t* sA = smem;
    uint8_t* sS = sA + C::kSmemA;
    float* stX = (float*)(sS + C::kSmemS);        // [128][K+4] At rows
    float* stY = stX + kTileM * C::kStageLd;      // [128][K+4] Bt rows
    uint64_t* bars = (uint64_t*)(stY + kTileM * C::kStageLd);
    uint64_t* full = bars;                        // TMA landed        (count 1 + tx)
    uint64_t* sready = bars + C::kStages;         // signs written     (count 2)
    uint64_t* empty = bars + 2 * C::kStages;      // MMAs done reading (count 1)
    uint64_t* tfull = bars + 3 * C::kStages;      // [2] accumulators ready
    uint64_t* tempty = tfull + 2;                 // [2] accumulators drained (count 4)
    uint64_t* mma_done = tempty + 2;
    uint64_t* red_go = mma_done + 1;              // leader -> member: write your partial (count 1)
    uint64_t* red_full = red_go + 1;              // members -> leader: partials written (count cs-1)
    uint32_t* tmem_slot = (uint32_t*)(red_full + 1);
    volatile int* abort = (volatile int*)(tmem_slot + 1);

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    if (threadIdx.x == 0) {
        for (int s = 0; s < C::kStages; ++s) {
            mbar_init(smem_u32(&full[s]), 1);
            mbar_init(smem_u32(&sready[s]), 2);
            mbar_init(smem_u32(&empty[s]), 1);
        }
        for (int b = 0; b < 2; ++b) {
            mbar_init(smem_u32(&tfull[b]), 1);
            mbar_init(smem_u32(&tempty[b]), 4);
        }
        mbar_init(smem_u32(mma_done), 1);
        mbar_init(smem_u32(red_go), 1);
        mbar_init(smem_u32(red_full), p.cs > 1 ? p.cs - 1 : 1);
        *abort = 0;
        fence_mbar_init();
    }
    if (warp == 1) {
        tmem_alloc(smem_u32(tmem_slot), C::kTmemCols);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    cluster_sync();  // every CTA's barriers exist before any remote arrive
    tc_fence_after();
    const uint32_t tmem = *tmem_slot;
    // examples are shared out per cluster; token tiles per CTA rank within it
    const uint32_t crank = cluster_rank(), cid = blockIdx.x / p.cs, ncl = gridDim.x / p.cs;

    const int nk_tot = p.nk_in + p.nk_out;
    if (warp == 0 && lane == 0) {
        // ---------------- TMA producer
        uint32_t last_par[16];
        bool issued[16];
        for (int s = 0; s < C::kStages; ++s) issued[s] = false;
        uint32_t ring = 0;
        bool ok = true;
        for (int64_t n = cid; ok && n < p.N; n += ncl)
            for (int tt = (int)crank; ok && tt < p.n_ttiles; tt += p.cs)
                for (int kc = 0; kc < nk_tot; ++kc, ++ring) {
                    const int s = ring % C::kStages;
                    const uint32_t ph = (ring / C::kStages) & 1u;
                    if (!wait_bounded(smem_u32(&empty[s]), ph ^ 1u, abort, p.err)) {
                        ok = false;
                        break;
                    }
                    const bool side_b = kc >= p.nk_in;
                    const int d0 = (side_b ? kc - p.nk_in : kc) * kChunkK;
                    mbar_arrive_tx(smem_u32(&full[s]), kTileBytes);
                    tma_load_3d(smem_u32(sA + (size_t)s * kTileBytes), side_b ? &tmB : &tmA, d0, tt * kTileM,
                                (int)n, smem_u32(&full[s]));
                    issued[s] = true;
                    last_par[s] = ph;
                }
        // drain: every issued copy must land before the CTA may exit
        for (int s = 0; s < C::kStages; ++s)
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
        uint32_t ring = 0, tile = 0;
        bool ok = true;
        const uint32_t idesc = idesc_bf16(kTileM, K);
        for (int64_t n = cid; ok && n < p.N; n += ncl)
            for (int tt = (int)crank; ok && tt < p.n_ttiles; tt += p.cs, ++tile) {
                const uint32_t b = tile & 1u, use = tile >> 1;
                if (!wait_bounded(smem_u32(&tempty[b]), (use & 1u) ^ 1u, abort, p.err)) {
                    ok = false;
                    break;
                }
                tc_fence_after();
                for (int kc = 0; kc < nk_tot; ++kc, ++ring) {
                    const int s = ring % C::kStages;
                    const uint32_t ph = (ring / C::kStages) & 1u;
                    if (!wait_bounded(smem_u32(&full[s]), ph, abort, p.err) ||
                        !wait_bounded(smem_u32(&sready[s]), ph, abort, p.err)) {
                        ok = false;
                        break;
                    }
                    tc_fence_after();
                    const bool side_b = kc >= p.nk_in;
                    const int kk = side_b ? kc - p.nk_in : kc;
                    const uint32_t d_tmem = tmem + b * C::kAccCols + (side_b ? K : 0);
                    const uint64_t ad = sw128_desc(smem_u32(sA + (size_t)s * kTileBytes));
                    const uint64_t bd = sw128_desc(smem_u32(sS + (size_t)s * C::kSignBytes));
#pragma unroll
                    for (int k = 0; k < kChunkK / 16; ++k)
                        mma_bf16(d_tmem, ad + 2 * k, bd + 2 * k, idesc, (kk > 0 || k > 0) ? 1u : 0u);
                    mma_commit(smem_u32(&empty[s]));
                }
                if (!ok) break;
                mma_commit(smem_u32(&tfull[b]));
            }
        // all MMAs this thread issued have completed once mma_done fires
        mma_commit(smem_u32(mma_done));
        const uint64_t t0 = global_ns();
        while (!mbar_try_wait(smem_u32(mma_done), 0))
            if (global_ns() - t0 > kTimeoutNs) {
                atomicOr(p.err, kErrTimeout);
                break;
            }
    } else if (warp == 2 || warp == 3) {
        // ---------------- sign generators (two warps, one half-row each)
        uint32_t ring = 0;
        bool ok = true;
        for (int64_t n = cid; ok && n < p.N; n += ncl)
            for (int tt = (int)crank; ok && tt < p.n_ttiles; tt += p.cs)
                for (int kc = 0; kc < nk_tot; ++kc, ++ring) {
                    const int s = ring % C::kStages;
                    const uint32_t ph = (ring / C::kStages) & 1u;
                    bool got = true;
                    if (lane == 0) got = wait_bounded(smem_u32(&empty[s]), ph ^ 1u, abort, p.err);
                    got = __shfl_sync(0xffffffffu, got, 0);
                    __syncwarp();
                    if (!got) {
                        ok = false;
                        break;
                    }
                    const bool side_b = kc >= p.nk_in;
                    const uint64_t key = side_b ? p.key_out : p.key_in;
                    const uint64_t rb = (uint64_t)(side_b ? kc - p.nk_in : kc);
                    uint8_t* tile = sS + (size_t)s * C::kSignBytes;
                    for (int col = lane; col < K; col += 32)
                        write_sign_half(tile, col, sign_word(key, (uint32_t)col, rb), warp - 2);
                    fence_proxy_async();
                    __syncwarp();
                    if (lane == 0) mbar_arrive(smem_u32(&sready[s]));
                }
    } else if (warp >= 4) {
        // ---------------- epilogue: TMEM -> shared -> Phi += Bt^T At
        const int q = warp & 3;          // TMEM lane quadrant of this warp
        const int et = threadIdx.x - 128;
        const int row = q * 32 + lane;   // token within the tile
        const int rg = et >> 3, cg = et & 7;
        uint32_t tile = 0, red_use = 0;
        bool stop = false;
        for (int64_t n = cid; !stop && n < p.N; n += ncl) {
            float acc[C::RB][C::CB];
#pragma unroll
            for (int a = 0; a < C::RB; ++a)
#pragma unroll
                for (int c = 0; c < C::CB; ++c) acc[a][c] = 0.f;
            for (int tt = (int)crank; tt < p.n_ttiles; tt += p.cs, ++tile) {
                const uint32_t b = tile & 1u, use = tile >> 1;
                bool got = true;
                if (lane == 0) got = wait_bounded(smem_u32(&tfull[b]), use & 1u, abort, p.err);
                got = __shfl_sync(0xffffffffu, got, 0);
                if (epi_any(!got)) {
                    stop = true;
                    break;
                }
                tc_fence_after();
                const uint32_t tbase = tmem + ((uint32_t)(q * 32) << 16) + b * C::kAccCols;
#pragma unroll
                for (int c0 = 0; c0 < 2 * K; c0 += 16) {
                    float v[16];
                    tmem_ld16(tbase + c0, v);
                    float* dst = c0 < K ? stX + row * C::kStageLd + c0 : stY + row * C::kStageLd + (c0 - K);
#pragma unroll
                    for (int i = 0; i < 16; i += 4)
                        *reinterpret_cast<float4*>(dst + i) = make_float4(v[i], v[i + 1], v[i + 2], v[i + 3]);
                }
                tc_fence_before();
                __syncwarp();
                if (lane == 0) mbar_arrive(smem_u32(&tempty[b]));
                epi_sync();
#pragma unroll 4
                for (int t = 0; t < kTileM; ++t) {
                    float y[C::RB], x[C::CB];
#pragma unroll
                    for (int a = 0; a < C::RB; ++a) y[a] = stY[t * C::kStageLd + rg * C::RB + a];
#pragma unroll
                    for (int c = 0; c < C::CB; ++c) x[c] = stX[t * C::kStageLd + cg * C::CB + c];
#pragma unroll
                    for (int a = 0; a < C::RB; ++a)
#pragma unroll
                        for (int c = 0; c < C::CB; ++c) acc[a][c] = fmaf(y[a], x[c], acc[a][c]);
                }
                epi_sync();
            }
            if (stop) break;
            if (p.cs > 1) {
                // Cluster reduction of the partial Phi blocks into the leader (rank
                // 0). The leader's staging buffer (free between tiles) receives
                // member r's partial at offset (r-1)*K*K, thread-major.
                constexpr int kPer = C::RB * C::CB;
                const uint32_t slot = smem_u32(stX) + (uint32_t)(et * kPer) * 4u;
                bool got = true;
                if (crank == 0) {
                    if (et == 0)
                        for (int r = 1; r < p.cs; ++r) mbar_arrive_remote(smem_u32(red_go), (uint32_t)r);
                    if (lane == 0) got = wait_bounded_cluster(smem_u32(red_full), red_use & 1u, abort, p.err);
                    got = __shfl_sync(0xffffffffu, got, 0);
                    if (epi_any(!got)) break;
                    for (int r = 1; r < p.cs; ++r) {
                        const float* part = stX + (r - 1) * K * K + et * kPer;
#pragma unroll
                        for (int a = 0; a < C::RB; ++a)
#pragma unroll
                            for (int c = 0; c < C::CB; ++c) acc[a][c] += part[a * C::CB + c];
                    }
                    epi_sync();  // partials consumed; staging free for the next tile
                } else {
                    if (lane == 0) got = wait_bounded_cluster(smem_u32(red_go), red_use & 1u, abort, p.err);
                    got = __shfl_sync(0xffffffffu, got, 0);
                    if (epi_any(!got)) break;
                    const uint32_t dst = map_rank(slot, 0) + (crank - 1) * (uint32_t)(K * K) * 4u;
#pragma unroll
                    for (int a = 0; a < C::RB; ++a)
#pragma unroll
                        for (int c = 0; c < C::CB; ++c) st_cluster_f32(dst + (uint32_t)(a * C::CB + c) * 4u, acc[a][c]);
                    fence_acq_rel_cluster();
                    epi_sync();
                    if (et == 0) mbar_arrive_remote(smem_u32(red_full), 0u);
                }
                ++red_use;
                if (crank != 0) continue;
            }
            float* out = p.phi + n * p.ld_phi;
#pragma unroll
            for (int a = 0; a < C::RB; ++a)
#pragma unroll
                for (int c = 0; c < C::CB; ++c)
                    out[(rg * C::RB + a) * K + cg * C::CB + c] = acc[a][c] * p.scale;
        }
    }

    tc_fence_before();
    __syncthreads();
    if (warp == 1) {
        tc_fence_after();
        tmem_dealloc(tmem, C::kTmemCols);
    }
    cluster_sync();  // no CTA leaves while a peer may still write to it
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

// 3-D map over X[N][T][d] (bf16): box 64 (d) x 128 (t) x 1 (example), 128B swizzle,
// out-of-range elements read as zero.
bool make_map(CUtensorMap* tm, const void* X, int64_t N, int64_t T, int64_t d) {
    EncodeTiledFn enc = encode_fn();
    if (!enc) return false;
    cuuint64_t dims[3] = {(cuuint64_t)d, (cuuint64_t)T, (cuuint64_t)N};
    cuuint64_t strides[2] = {(cuuint64_t)(d * 2), (cuuint64_t)(T * d * 2)};
    cuuint32_t box[3] = {kChunkK, kTileM, 1};
    cuuint32_t estr[3] = {1, 1, 1};
    return enc(tm, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(X), dims, strides, box, estr,
               CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
               CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

bool device_is_sm103() {
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return false;
    int major = 0, minor = 0;
    cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev);
    cudaDeviceGetAttribute(&minor, cudaDevAttrComputeCapabilityMinor, dev);
    return major == 10 && minor == 3;
}

template <int K>
cudaError_t launch_k(const tda_layer_desc& L, const void* A, const void* B, int64_t N, float* phi,
                     int64_t ld_phi, unsigned int* err, cudaStream_t s) {
    using C = Cfg<K>;
    CUtensorMap tmA, tmB;
    if (!make_map(&tmA, A, N, L.T, L.d_in) || !make_map(&tmB, B, N, L.T, L.d_out)) return cudaErrorInvalidValue;
    Params p;
    p.N = N;
    p.T = L.T;
    p.d_in = L.d_in;
    p.d_out = L.d_out;
    p.ld_phi = ld_phi;
    p.key_in = side_key(L.seed, L.layer, 0);
    p.key_out = side_key(L.seed, L.layer, 1);
    p.scale = projection_scale(L);
    p.phi = phi;
    p.err = err;
    p.n_ttiles = (int)((L.T + kTileM - 1) / kTileM);
    p.nk_in = (int)((L.d_in + kChunkK - 1) / kChunkK);
    p.nk_out = (int)((L.d_out + kChunkK - 1) / kChunkK);
    static int sms = 0;
    if (!sms) {
        int dev = 0;
        cudaGetDevice(&dev);
        cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
        if (sms <= 0) sms = 1;
    }
    cudaError_t e = cudaFuncSetAttribute(project_tc_kernel<K>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         (int)C::kSmem);
    if (e != cudaSuccess) return e;
    // Fewer examples than SMs: a cluster of cs CTAs shares each example's token
    // tiles and reduces the partial features through distributed shared memory.
    int cs = 1;
    if (N < sms) cs = (2 * N >= sms) ? 2 : 4;
    while (cs > 1 && cs > p.n_ttiles) cs >>= 1;
    p.cs = cs;
    cudaLaunchConfig_t cfg = {};
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = (unsigned)cs;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    cfg.blockDim = dim3(kThreads);
    cfg.dynamicSmemBytes = C::kSmem;
    cfg.stream = s;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    int64_t clusters = N;
    int max_clusters = 0;
    cfg.gridDim = dim3((unsigned)(cs * (sms / cs)));
    if (cudaOccupancyMaxActiveClusters(&max_clusters, project_tc_kernel<K>, &cfg) != cudaSuccess || max_clusters < 1)
        max_clusters = sms / cs;
    if (clusters > max_clusters) clusters = max_clusters;
    cfg.gridDim = dim3((unsigned)(clusters * cs));
    note_launches(1);
    e = cudaLaunchKernelEx(&cfg, project_tc_kernel<K>, tmA, tmB, p);
    if (e != cudaSuccess) return e;
    return cudaGetLastError();
}

}  // namespace

bool project_tc_supported(const tda_layer_desc& L, const void* A, const void* B) {
    static int sm103 = -1;
    if (sm103 < 0) sm103 = device_is_sm103() ? 1 : 0;
    if (!sm103 || !encode_fn()) return false;
    if (L.kind != TDA_PROJ_RADEMACHER || L.k_in != L.k_out) return false;
    if (L.k_in != 16 && L.k_in != 32 && L.k_in != 64) return false;
    if (L.d_in % 8 || L.d_out % 8 || L.T < 1) return false;
    if (((uintptr_t)A & 15) || ((uintptr_t)B & 15)) return false;
    if (L.T > (1LL << 30) || L.d_in > (1LL << 30) || L.d_out > (1LL << 30)) return false;
    return true;
}

cudaError_t launch_project_tc(const tda_layer_desc& L, const void* A, const void* B, int64_t N, float* phi,
                              int64_t ld_phi, unsigned int* err, cudaStream_t s) {
    if (N == 0) return cudaSuccess;
    switch (L.k_in) {
        case 16: return launch_k<16>(L, A, B, N, phi, ld_phi, err, s);
        case 32: return launch_k<32>(L, A, B, N, phi, ld_phi, err, s);
        case 64: return launch_k<64>(L, A, B, N, phi, ld_phi, err, s);
        default: return cudaErrorNotSupported;
    }
}

}  // namespace tda
