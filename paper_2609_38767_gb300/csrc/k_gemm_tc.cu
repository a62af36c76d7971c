// k_gemm_tc.cu -- the score GEMM on the 5th-generation tensor cores:
//   S[n][m] = beta * S[n][m] + sum_k Phi[m][k] * Qhat[n][k]
// (gradient inner products between training features Phi and preconditioned
// query features Qhat, Sec. 3.2 / Eq. 4's left side) for fp32 operands.
//
// fp32 accuracy from TF32 tensor cores ("3xTF32"): every operand x is split as
// x = hi + lo with hi = x truncated to TF32 (exact) and lo = x - hi (exact in
// fp32); the product is hi*hi' + hi*lo' + lo*hi', dropping lo*lo' (relative
// size ~2^-22). Each K=8 step therefore issues three tcgen05.mma.kind::tf32.
//
// CTA tile: 128 rows of Phi (MMA M, one TMEM lane each) x BN query columns
// (MMA N). Lane 0 of warp 5 copies the fp32 chunks of both operands with TMA
// (32 features = one 128-byte row per operand row, 128B swizzle: already the
// K-major operand layout) into the hi tiles of a stage; warps 0-3 write lo to
// the lo tile at the same offset (the fp32 tile itself is the hi operand: a
// kind::tf32 MMA reads only the upper 19 bits); lane 0 of warp 4 issues the
// MMAs; warps 4-7 read the fp32 accumulator tile from TMEM. A thread-block
// cluster of cs CTAs splits K; the members' partial tiles are summed into the
// leader CTA over distributed shared memory (deterministic, no workspace)
// before the leader writes S. With more tiles than SMs and short K (the blocked
// Cholesky's products) gemm3x_persist_kernel walks the tiles instead. All
// waits are bounded (see tc_ptx.cuh).
#include <cuda.h>

#include <mutex>

#include "tda_internal.cuh"

namespace tda {
namespace {

#include "tc_ptx.cuh"

constexpr int kThreads = 256;
constexpr int kBM = 128;       // Phi rows per tile
constexpr int kKC = 32;        // fp32 elements per K chunk (one 128-byte operand row)
constexpr uint32_t kRowBytes = kKC * 4;

template <int BN>
struct GCfg {
    static constexpr int kStages = BN <= 64 ? 4 : (BN <= 128 ? 3 : 2);
    static constexpr uint32_t kABytes = kBM * kRowBytes;   // 16 KiB
    static constexpr uint32_t kBBytes = BN * kRowBytes;
    static constexpr uint32_t kStageBytes = 2 * kABytes + 2 * kBBytes;  // hi and lo of both operands
    // K chunks rotate over kAcc accumulators (all 512 TMEM columns): each sees
    // 1/kAcc of the additions, which bounds the tensor core's fp32 accumulation
    // error; the epilogue sums them on CUDA cores with round-to-nearest.
    static constexpr int kAcc = 512 / BN < 8 ? 512 / BN : 8;
    static constexpr uint32_t kTmemCols = 512;
    static constexpr size_t kSmem = 1024 + (size_t)kStages * kStageBytes + 8 * (3 * kStages + 4) + 16;  // + barriers, TMEM slot, abort flag
};

struct GParams {
    const float* A;  // Phi, n_t rows
    const float* B;  // Qhat, n_q rows
    float* S;
    int64_t n_t, n_q, K, lda, ldb, ld_S;
    float beta, alpha;     // S = beta * S + alpha * (product); the score uses alpha = 1
    int lower;             // square product (n_t == n_q, BN == kBM): only tiles with m0 <= n0
    int cs, tiles_n;
    int64_t kslice, slab;  // split-K over gridDim.y: K slice per CTA row, S stride per slice (0: no split)
    int splits;            // gridDim.y
    int batched;           // grid z = batch entry: A and B maps are 3-D (z the third coordinate)
    int64_t s_z;           // S element offset between batch entries
    int64_t tiles_z;       // persistent kernel: tiles per batch entry
    int nz;                // persistent kernel: batch entries
    unsigned int* err;
};

// Instruction descriptor, kind::tf32: tf32 A and B (format 2), fp32 D, both K-major.
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

// Split a TMA-written fp32 tile: lo = x - hi (hi = x truncated to TF32) goes to
// the lo tile at the same byte offset (the swizzle is the same for both). The
// fp32 tile itself serves as the hi operand: a kind::tf32 MMA reads only the
// upper 19 bits of each element, which is hi exactly, so it is not rewritten.
// 128 threads, one 16-byte group each per pass (conflict-free).
template <uint32_t BYTES>
__device__ __forceinline__ void split_tile(const uint8_t* hi, uint8_t* lo, int pt) {
#pragma unroll 4
    for (uint32_t off = (uint32_t)pt * 16u; off < BYTES; off += 128u * 16u) {
        const float4 v = *reinterpret_cast<const float4*>(hi + off);
        float4 h, l;
        split_tf32(v.x, h.x, l.x);
        split_tf32(v.y, h.y, l.y);
        split_tf32(v.z, h.z, l.z);
        split_tf32(v.w, h.w, l.w);
        *reinterpret_cast<float4*>(lo + off) = l;
    }
}
__device__ __forceinline__ void tma_load_2d(uint32_t dst, const CUtensorMap* tm, int c0, int c1, uint32_t bar) {
    asm volatile(
        "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3}], [%4];" ::"r"(
            dst),
        "l"((uint64_t)tm), "r"(c0), "r"(c1), "r"(bar)
        : "memory");
}

template <int BN>
__global__ void __launch_bounds__(kThreads, 1)
score3x_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB, const GParams p) {
    using C = GCfg<BN>;
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = (uint8_t*)(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
    uint64_t* bars = (uint64_t*)(smem + (size_t)C::kStages * C::kStageBytes);
    uint64_t* full = bars;                   // count 4 (producer warps)
    uint64_t* empty = bars + C::kStages;     // count 1 (MMA commit)
    uint64_t* tfull = empty + C::kStages;    // count 1
    uint64_t* red_go = tfull + 1;            // count 1 (leader's remote arrive)
    uint64_t* red_full = red_go + 1;         // count cs-1
    uint64_t* mma_done = red_full + 1;       // count 1
    uint64_t* raw_full = mma_done + 1;       // [kStages] TMA bytes landed (count 1 + tx)
    uint32_t* tmem_slot = (uint32_t*)(raw_full + C::kStages);
    volatile int* abort = (volatile int*)(tmem_slot + 1);

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    if (threadIdx.x == 0) {
        for (int s = 0; s < C::kStages; ++s) {
            mbar_init(smem_u32(&full[s]), 4);
            mbar_init(smem_u32(&empty[s]), 1);
            mbar_init(smem_u32(&raw_full[s]), 1);
        }
        mbar_init(smem_u32(tfull), 1);
        mbar_init(smem_u32(red_go), 1);
        mbar_init(smem_u32(red_full), p.cs > 1 ? p.cs - 1 : 1);
        mbar_init(smem_u32(mma_done), 1);
        *abort = 0;
        fence_mbar_init();
    }
    if (warp == 4) {
        tmem_alloc(smem_u32(tmem_slot), C::kTmemCols);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    cluster_sync();
    tc_fence_after();
    const uint32_t tmem = *tmem_slot;

    const uint32_t crank = cluster_rank();
    const int64_t tile = blockIdx.x / p.cs;
    int64_t m0 = (tile / p.tiles_n) * kBM, n0 = (tile % p.tiles_n) * BN;
    if (p.lower) {
        // tile t of the lower triangle: row tile i (n), column tile j (m) <= i, t = i(i+1)/2 + j
        int64_t i = (int64_t)((sqrt(8.0 * (double)tile + 1.0) - 1.0) * 0.5);
        while (i * (i + 1) / 2 > tile) --i;
        while ((i + 1) * (i + 2) / 2 <= tile) ++i;
        n0 = i * BN;
        m0 = (tile - i * (i + 1) / 2) * kBM;
    }
    // split-K slice z covers features [z*kslice, z*kslice + Kz) and writes its own slab of S
    const int64_t kbase = (int64_t)blockIdx.y * p.kslice;
    const int64_t Kz = p.kslice ? ((p.K - kbase) < p.kslice ? (p.K - kbase) : p.kslice) : p.K;
    float* Sz = p.S + (int64_t)blockIdx.y * p.slab + (int64_t)blockIdx.z * p.s_z;
    const int zc = (int)blockIdx.z;
    const int64_t nkc = (Kz + kKC - 1) / kKC;
    const int64_t per = (nkc + p.cs - 1) / p.cs;
    const int64_t kc0 = crank * per, kc1 = (kc0 + per) < nkc ? (kc0 + per) : nkc;

    if (warp < 4) {
        // ---------------- split warps: raw fp32 (TMA) -> hi in place + lo
        const int pt = threadIdx.x;
        uint32_t it = 0;
        for (int64_t kc = kc0; kc < kc1; ++kc, ++it) {
            const int s = it % C::kStages;
            const uint32_t ph = (it / C::kStages) & 1u;
            bool got = true;
            if (lane == 0) got = wait_bounded(smem_u32(&raw_full[s]), ph, abort, p.err);
            got = __shfl_sync(0xffffffffu, got, 0);
            __syncwarp();
            if (!got) break;
            uint8_t* st = smem + (size_t)s * C::kStageBytes;
            split_tile<C::kABytes>(st, st + C::kABytes, pt);
            split_tile<C::kBBytes>(st + 2 * C::kABytes, st + 2 * C::kABytes + C::kBBytes, pt);
            fence_proxy_async();
            __syncwarp();
            if (lane == 0) mbar_arrive(smem_u32(&full[s]));
        }
    } else {
        if (warp == 5 && lane == 0) {
            // ---------------- TMA producer: fp32 chunks of Phi rows m0.. and Qhat rows n0..
            // (features past the slice end belong to the next slice only when the slice
            // is not the last; slices are multiples of 32 features, so no chunk crosses one)
            uint32_t it = 0, last_par[C::kStages];
            bool issued[C::kStages];
            for (int s = 0; s < C::kStages; ++s) issued[s] = false;
            for (int64_t kc = kc0; kc < kc1; ++kc, ++it) {
                const int s = it % C::kStages;
                const uint32_t ph = (it / C::kStages) & 1u;
                if (!wait_bounded(smem_u32(&empty[s]), ph ^ 1u, abort, p.err)) break;
                const uint32_t st = smem_u32(smem + (size_t)s * C::kStageBytes), bar = smem_u32(&raw_full[s]);
                const int k = (int)(kbase + kc * kKC);
                mbar_arrive_tx(bar, C::kABytes + C::kBBytes);
                if (p.batched) {
                    tma_load_3d(st, &tmA, k, (int)m0, zc, bar);
                    tma_load_3d(st + 2 * C::kABytes, &tmB, k, (int)n0, zc, bar);
                } else {
                    tma_load_2d(st, &tmA, k, (int)m0, bar);
                    tma_load_2d(st + 2 * C::kABytes, &tmB, k, (int)n0, bar);
                }
                issued[s] = true;
                last_par[s] = ph;
            }
            // copies still in flight when the consumers stopped early land before the CTA exits
            for (int s = 0; s < C::kStages; ++s)
                if (issued[s]) {
                    const uint64_t t0 = global_ns();
                    while (!mbar_try_wait(smem_u32(&raw_full[s]), last_par[s]))
                        if (global_ns() - t0 > kTimeoutNs) {
                            atomicOr(p.err, kErrTimeout);
                            break;
                        }
                }
        }
        if (warp == 4 && lane == 0) {
            // ---------------- MMA issuer
            const uint32_t idesc = idesc_tf32(kBM, BN);
            uint32_t it = 0;
            bool ok = true;
            for (int64_t kc = kc0; kc < kc1; ++kc, ++it) {
                const int s = it % C::kStages;
                const uint32_t ph = (it / C::kStages) & 1u;
                if (!wait_bounded(smem_u32(&full[s]), ph, abort, p.err)) {
                    ok = false;
                    break;
                }
                tc_fence_after();
                const uint32_t st = smem_u32(smem + (size_t)s * C::kStageBytes);
                const uint64_t ahi = sw128_desc(st), alo = sw128_desc(st + C::kABytes);
                const uint64_t bhi = sw128_desc(st + 2 * C::kABytes), blo = sw128_desc(st + 2 * C::kABytes + C::kBBytes);
#pragma unroll
                for (int k = 0; k < kKC / 8; ++k) {  // K = 8 tf32 = 32 bytes per instruction
                    const uint32_t d = tmem + (it % C::kAcc) * BN;
                    const uint32_t first = (it < (uint32_t)C::kAcc && k == 0) ? 0u : 1u;
                    mma_tf32(d, ahi + 2 * k, bhi + 2 * k, idesc, first);
                    mma_tf32(d, ahi + 2 * k, blo + 2 * k, idesc, 1u);
                    mma_tf32(d, alo + 2 * k, bhi + 2 * k, idesc, 1u);
                }
                mma_commit(smem_u32(&empty[s]));
            }
            if (ok) mma_commit(smem_u32(tfull));
            mma_commit(smem_u32(mma_done));
            const uint64_t t0 = global_ns();
            while (!mbar_try_wait(smem_u32(mma_done), 0))
                if (global_ns() - t0 > kTimeoutNs) {
                    atomicOr(p.err, kErrTimeout);
                    break;
                }
        }
        __syncwarp();
        // ---------------- epilogue (warps 4-7): TMEM -> (cluster reduction) -> S
        const int q = warp & 3;
        const int row = q * 32 + lane;  // Phi row within the tile
        const bool empty_k = kc1 <= kc0;
        bool got = true;
        if (!empty_k) {
            if (lane == 0) got = wait_bounded(smem_u32(tfull), 0, abort, p.err);
            got = __shfl_sync(0xffffffffu, got, 0);
        }
        float acc[BN];
        if (!epi_any(!got)) {
            tc_fence_after();
            const uint32_t tbase = tmem + ((uint32_t)(q * 32) << 16);
            const int used = (int)((kc1 - kc0) < C::kAcc ? (kc1 - kc0) : C::kAcc);  // accumulators written
#pragma unroll
            for (int c0 = 0; c0 < BN; c0 += 16) {
#pragma unroll
                for (int i = 0; i < 16; ++i) acc[c0 + i] = 0.f;
                for (int a = 0; a < used; ++a) {
                    float v[16];
                    tmem_ld16(tbase + a * BN + c0, v);
#pragma unroll
                    for (int i = 0; i < 16; ++i) acc[c0 + i] += v[i];
                }
            }
            tc_fence_before();
            bool ok = true;
            if (p.cs > 1) {
                // partial tiles of members 1..cs-1 land in the leader's stage buffers
                float* red = (float*)smem;
                const uint32_t slot = smem_u32(red) + (uint32_t)(row * BN) * 4u;
                if (crank == 0) {
                    if (threadIdx.x == 128)
                        for (int r = 1; r < p.cs; ++r) mbar_arrive_remote(smem_u32(red_go), (uint32_t)r);
                    bool g2 = true;
                    if (lane == 0) g2 = wait_bounded_cluster(smem_u32(red_full), 0, abort, p.err);
                    g2 = __shfl_sync(0xffffffffu, g2, 0);
                    ok = !epi_any(!g2);
                    if (ok)
                        for (int r = 1; r < p.cs; ++r) {
                            const float* part = red + (size_t)(r - 1) * kBM * BN + (size_t)row * BN;
#pragma unroll
                            for (int c = 0; c < BN; c += 4) {
                                const float4 v = *reinterpret_cast<const float4*>(part + c);
                                acc[c] += v.x;
                                acc[c + 1] += v.y;
                                acc[c + 2] += v.z;
                                acc[c + 3] += v.w;
                            }
                        }
                } else {
                    bool g2 = true;
                    if (lane == 0) g2 = wait_bounded_cluster(smem_u32(red_go), 0, abort, p.err);
                    g2 = __shfl_sync(0xffffffffu, g2, 0);
                    ok = !epi_any(!g2);
                    if (ok) {
                        const uint32_t dst = map_rank(slot, 0) + (crank - 1) * (uint32_t)(kBM * BN) * 4u;
#pragma unroll
                        for (int c = 0; c < BN; ++c) st_cluster_f32(dst + (uint32_t)c * 4u, acc[c]);
                        fence_acq_rel_cluster();
                        epi_sync();
                        if (threadIdx.x == 128) mbar_arrive_remote(smem_u32(red_full), 0u);
                    }
                    ok = false;  // members write nothing to S
                }
            }
            if (ok) {
                const int64_t m = m0 + row;
                if (m < p.n_t) {
                    if (p.beta == 0.f) {
#pragma unroll
                        for (int c = 0; c < BN; ++c) {
                            const int64_t n = n0 + c;
                            if (n < p.n_q) Sz[n * p.ld_S + m] = p.alpha * acc[c];
                        }
                    } else {
                        // the previous values of 32 columns are loaded before any is stored, so
                        // the loads are in flight together instead of one round trip per column
#pragma unroll
                        for (int c0 = 0; c0 < BN; c0 += 32) {
                            float old[32];
#pragma unroll
                            for (int i = 0; i < 32; ++i) {
                                const int64_t n = n0 + c0 + i;
                                old[i] = n < p.n_q ? __ldcg(Sz + n * p.ld_S + m) : 0.f;
                            }
#pragma unroll
                            for (int i = 0; i < 32; ++i) {
                                const int64_t n = n0 + c0 + i;
                                if (n < p.n_q) Sz[n * p.ld_S + m] = p.beta * old[i] + p.alpha * acc[c0 + i];
                            }
                        }
                    }
                }
            }
        }
    }

    tc_fence_before();
    __syncthreads();
    if (warp == 4) {
        tc_fence_after();
        tmem_dealloc(tmem, C::kTmemCols);
    }
    cluster_sync();
}

// ---------------------------------------------------------------------------
// Persistent variant of the same product for many tiles with short K (the
// blocked Cholesky's trailing updates and the substitutions' block products,
// K = 128 or 256): each CTA walks tiles blockIdx.x, blockIdx.x + gridDim.x, ...
// over all batch entries with one set of barriers and one TMEM allocation. The
// accumulators are double-buffered (kAcc per buffer), so a tile's epilogue
// (TMEM -> registers -> S) overlaps the next tile's loads, splits and MMAs.
// Warps 0-3 split, warps 4-7 epilogue, lane 0 of warp 8 issues the TMA copies,
// lane 0 of warp 9 the MMAs. Same arithmetic per tile as score3x_kernel (the
// K chunks rotate over kAcc accumulators, summed on CUDA cores). No clusters,
// no split-K. All waits are bounded. Ten warps share the register file's four
// partitions unevenly (three warps on two of them), which caps a thread at 168
// registers: the epilogue drains the accumulators 64 columns at a time.
constexpr int kThreadsP = 320;

template <int BN>
struct PCfg {
    static constexpr int kStages = GCfg<BN>::kStages;
    static constexpr uint32_t kABytes = GCfg<BN>::kABytes;
    static constexpr uint32_t kBBytes = GCfg<BN>::kBBytes;
    static constexpr uint32_t kStageBytes = GCfg<BN>::kStageBytes;
    static constexpr int kAcc = 256 / BN;  // per buffer: two buffers fill the 512 TMEM columns
    static constexpr size_t kSmem = 1024 + (size_t)kStages * kStageBytes + 8 * (3 * kStages + 5) + 16;
};

// Rows m0 (of A) and n0 (of B) and batch entry z of tile t.
template <int BN>
__device__ __forceinline__ void tile_at(const GParams& p, int64_t t, int64_t& m0, int64_t& n0, int& z) {
    z = (int)(t / p.tiles_z);
    const int64_t tile = t - (int64_t)z * p.tiles_z;
    if (p.lower) {
        int64_t i = (int64_t)((sqrt(8.0 * (double)tile + 1.0) - 1.0) * 0.5);
        while (i * (i + 1) / 2 > tile) --i;
        while ((i + 1) * (i + 2) / 2 <= tile) ++i;
        n0 = i * BN;
        m0 = (tile - i * (i + 1) / 2) * kBM;
    } else {
        m0 = (tile / p.tiles_n) * kBM;
        n0 = (tile % p.tiles_n) * BN;
    }
}

template <int BN>
__global__ void __launch_bounds__(kThreadsP, 1)
gemm3x_persist_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
                      const GParams p) {
    using C = PCfg<BN>;
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = (uint8_t*)(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
    uint64_t* bars = (uint64_t*)(smem + (size_t)C::kStages * C::kStageBytes);
    uint64_t* raw_full = bars;                  // [kStages] TMA bytes landed (count 1 + tx)
    uint64_t* full = raw_full + C::kStages;     // [kStages] split into hi/lo (count 4)
    uint64_t* empty = full + C::kStages;        // [kStages] MMAs done reading (count 1)
    uint64_t* tfull = empty + C::kStages;       // [2] accumulators ready (count 1)
    uint64_t* tempty = tfull + 2;               // [2] accumulators drained (count 4)
    uint64_t* mma_done = tempty + 2;            // count 1
    uint32_t* tmem_slot = (uint32_t*)(mma_done + 1);
    volatile int* abort = (volatile int*)(tmem_slot + 1);

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    if (threadIdx.x == 0) {
        for (int s = 0; s < C::kStages; ++s) {
            mbar_init(smem_u32(&raw_full[s]), 1);
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
    if (warp == 9) {
        tmem_alloc(smem_u32(tmem_slot), 512);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *tmem_slot;
    const int64_t total = p.tiles_z * p.nz;
    const int64_t nkc = (p.K + kKC - 1) / kKC;

    if (warp < 4) {
        // ---------------- split warps: raw fp32 (TMA) -> hi in place + lo
        const int pt = threadIdx.x;
        uint32_t it = 0;
        bool ok = true;
        for (int64_t t = blockIdx.x; ok && t < total; t += gridDim.x)
            for (int64_t kc = 0; kc < nkc; ++kc, ++it) {
                const int s = it % C::kStages;
                const uint32_t ph = (it / C::kStages) & 1u;
                bool got = true;
                if (lane == 0) got = wait_bounded(smem_u32(&raw_full[s]), ph, abort, p.err);
                got = __shfl_sync(0xffffffffu, got, 0);
                __syncwarp();
                if (!got) {
                    ok = false;
                    break;
                }
                uint8_t* st = smem + (size_t)s * C::kStageBytes;
                split_tile<C::kABytes>(st, st + C::kABytes, pt);
                split_tile<C::kBBytes>(st + 2 * C::kABytes, st + 2 * C::kABytes + C::kBBytes, pt);
                fence_proxy_async();
                __syncwarp();
                if (lane == 0) mbar_arrive(smem_u32(&full[s]));
            }
    } else if (warp < 8) {
        // ---------------- epilogue: TMEM -> registers (buffer released) -> S
        const int q = warp & 3;
        const int row = q * 32 + lane;
        const int used = (int)(nkc < C::kAcc ? nkc : C::kAcc);
        uint32_t lt = 0;
        for (int64_t t = blockIdx.x; t < total; t += gridDim.x, ++lt) {
            const uint32_t b = lt & 1u, ph = (lt >> 1) & 1u;
            bool got = true;
            if (lane == 0) got = wait_bounded(smem_u32(&tfull[b]), ph, abort, p.err);
            got = __shfl_sync(0xffffffffu, got, 0);
            if (epi_any(!got)) break;
            tc_fence_after();
            const uint32_t tbase = tmem + ((uint32_t)(q * 32) << 16) + b * (uint32_t)(C::kAcc * BN);
            int64_t m0, n0;
            int z;
            tile_at<BN>(p, t, m0, n0, z);
            float* Sz = p.S + (int64_t)z * p.s_z;
            const int64_t m = m0 + row;
            // 64 columns at a time (register budget): the part's previous values are loaded first,
            // so the 64 loads are in flight while the part's accumulators are read from TMEM; the
            // buffer is released after the last read
            constexpr int HW = BN < 64 ? BN : 64;
            const bool rmw = p.beta != 0.f && m < p.n_t;
#pragma unroll 1
            for (int h0 = 0; h0 < BN; h0 += HW) {
                float old[HW];
                if (rmw) {
#pragma unroll
                    for (int i = 0; i < HW; ++i) {
                        const int64_t n = n0 + h0 + i;
                        old[i] = n < p.n_q ? __ldcg(Sz + n * p.ld_S + m) : 0.f;
                    }
                }
                float acc[HW];
#pragma unroll
                for (int c0 = 0; c0 < HW; c0 += 16) {
#pragma unroll
                    for (int i = 0; i < 16; ++i) acc[c0 + i] = 0.f;
                    for (int a = 0; a < used; ++a) {
                        float v[16];
                        tmem_ld16(tbase + a * BN + h0 + c0, v);
#pragma unroll
                        for (int i = 0; i < 16; ++i) acc[c0 + i] += v[i];
                    }
                }
                if (h0 + HW >= BN) {
                    tc_fence_before();
                    __syncwarp();
                    if (lane == 0) mbar_arrive(smem_u32(&tempty[b]));
                }
                if (m < p.n_t) {
#pragma unroll
                    for (int i = 0; i < HW; ++i) {
                        const int64_t n = n0 + h0 + i;
                        if (n < p.n_q) Sz[n * p.ld_S + m] = rmw ? p.beta * old[i] + p.alpha * acc[i] : p.alpha * acc[i];
                    }
                }
            }
        }
    } else if (warp == 8 && lane == 0) {
        // ---------------- TMA producer
        uint32_t it = 0, last_par[C::kStages];
        bool issued[C::kStages];
        for (int s = 0; s < C::kStages; ++s) issued[s] = false;
        bool ok = true;
        for (int64_t t = blockIdx.x; ok && t < total; t += gridDim.x) {
            int64_t m0, n0;
            int z;
            tile_at<BN>(p, t, m0, n0, z);
            for (int64_t kc = 0; kc < nkc; ++kc, ++it) {
                const int s = it % C::kStages;
                const uint32_t ph = (it / C::kStages) & 1u;
                if (!wait_bounded(smem_u32(&empty[s]), ph ^ 1u, abort, p.err)) {
                    ok = false;
                    break;
                }
                const uint32_t st = smem_u32(smem + (size_t)s * C::kStageBytes), bar = smem_u32(&raw_full[s]);
                const int k = (int)(kc * kKC);
                mbar_arrive_tx(bar, C::kABytes + C::kBBytes);
                if (p.batched) {
                    tma_load_3d(st, &tmA, k, (int)m0, z, bar);
                    tma_load_3d(st + 2 * C::kABytes, &tmB, k, (int)n0, z, bar);
                } else {
                    tma_load_2d(st, &tmA, k, (int)m0, bar);
                    tma_load_2d(st + 2 * C::kABytes, &tmB, k, (int)n0, bar);
                }
                issued[s] = true;
                last_par[s] = ph;
            }
        }
        for (int s = 0; s < C::kStages; ++s)
            if (issued[s]) {
                const uint64_t t0 = global_ns();
                while (!mbar_try_wait(smem_u32(&raw_full[s]), last_par[s]))
                    if (global_ns() - t0 > kTimeoutNs) {
                        atomicOr(p.err, kErrTimeout);
                        break;
                    }
            }
    } else if (warp == 9 && lane == 0) {
        // ---------------- MMA issuer
        const uint32_t idesc = idesc_tf32(kBM, BN);
        uint32_t it = 0, lt = 0;
        bool ok = true;
        for (int64_t t = blockIdx.x; ok && t < total; t += gridDim.x, ++lt) {
            const uint32_t b = lt & 1u, use = lt >> 1;
            if (!wait_bounded(smem_u32(&tempty[b]), (use & 1u) ^ 1u, abort, p.err)) break;
            tc_fence_after();
            for (int64_t kc = 0; kc < nkc; ++kc, ++it) {
                const int s = it % C::kStages;
                const uint32_t ph = (it / C::kStages) & 1u;
                if (!wait_bounded(smem_u32(&full[s]), ph, abort, p.err)) {
                    ok = false;
                    break;
                }
                tc_fence_after();
                const uint32_t st = smem_u32(smem + (size_t)s * C::kStageBytes);
                const uint64_t ahi = sw128_desc(st), alo = sw128_desc(st + C::kABytes);
                const uint64_t bhi = sw128_desc(st + 2 * C::kABytes), blo = sw128_desc(st + 2 * C::kABytes + C::kBBytes);
                const uint32_t d = tmem + (b * C::kAcc + (uint32_t)(kc % C::kAcc)) * BN;
#pragma unroll
                for (int k = 0; k < kKC / 8; ++k) {
                    const uint32_t first = (kc < C::kAcc && k == 0) ? 0u : 1u;
                    mma_tf32(d, ahi + 2 * k, bhi + 2 * k, idesc, first);
                    mma_tf32(d, ahi + 2 * k, blo + 2 * k, idesc, 1u);
                    mma_tf32(d, alo + 2 * k, bhi + 2 * k, idesc, 1u);
                }
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

    tc_fence_before();
    __syncthreads();
    if (warp == 9) {
        tc_fence_after();
        tmem_dealloc(tmem, 512);
    }
}

// ---------------------------------------------------------------------------
// Fisher fit on the tensor cores: M_l += Phi_l^T Phi_l for the lower 128 x 128
// tiles of every layer l (layer l's features at column l*D of each row of Phi).
// The MMA operand tiles are features x examples, K-major (32 examples per
// chunk), but Phi holds examples x features. Lane 0 of warp 5 copies each chunk
// raw with TMA (32 examples x 32 features per box, 128-byte swizzle, 4 boxes
// per operand) into a ring of raw stages; warps 0-3 read it back transposed
// (lane = example, 16 bytes of features per load: conflict-free thanks to the
// swizzle), split every value to hi/lo and write both into the K-major swizzled
// operand layout (conflict-free: the 32 lanes hit 32 distinct banks). A tile on
// the diagonal has A = B and loads and splits one operand.
template <int ROWS>
__device__ __forceinline__ void store_split_t(const float4 (&vals)[ROWS / 16], uint8_t* hi, uint8_t* lo, int pt) {
    constexpr int kPer = ROWS / 16;
    const int lane = pt & 31, w = pt >> 5;
#pragma unroll
    for (int j = 0; j < kPer; ++j) {
        const float in[4] = {vals[j].x, vals[j].y, vals[j].z, vals[j].w};
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            const int fr = (ROWS / 4) * w + 4 * j + i;  // feature row of the tile
            const uint32_t off = (uint32_t)fr * kRowBytes + (uint32_t)((((lane >> 2) ^ (fr & 7)) << 4) + (lane & 3) * 4);
            float h, l;
            split_tf32(in[i], h, l);
            *reinterpret_cast<float*>(hi + off) = h;
            *reinterpret_cast<float*>(lo + off) = l;
        }
    }
}
// Warp w's 32 features of one raw operand (box w: row = example, 128 bytes of
// features, 16-byte groups swizzled by the row's low three bits).
__device__ __forceinline__ void load_raw_t(const uint8_t* raw, float4 (&vals)[8], int pt) {
    const int lane = pt & 31, w = pt >> 5;
    const uint8_t* row = raw + (uint32_t)w * 4096u + (uint32_t)lane * kRowBytes;
#pragma unroll
    for (int j = 0; j < 8; ++j) vals[j] = *reinterpret_cast<const float4*>(row + ((j ^ (lane & 7)) << 4));
}

struct FCfg {
    static constexpr int kStages = 2;       // hi/lo operand stages
    static constexpr int kRawStages = 3;    // raw TMA chunks
    static constexpr uint32_t kABytes = kBM * kRowBytes;    // 16 KiB: one operand, hi or lo or raw
    static constexpr uint32_t kStageBytes = 4 * kABytes;    // hi and lo of both operands
    static constexpr uint32_t kRawBytes = 2 * kABytes;      // raw chunk of both operands
    // The tensor pipe's fp32 accumulation rounds toward zero, so a long same-sign sum
    // (a diagonal entry of M) drifts low by ~1 ulp per accumulate. Each accumulator
    // therefore takes a group of kGroup consecutive chunks (48 accumulates) and the
    // epilogue warps drain it into round-to-nearest fp32 registers while the MMAs
    // move on to the next of the kAcc accumulators.
    static constexpr int kAcc = 4;                          // 4 x 128 TMEM columns
    static constexpr int kGroup = 4;                        // chunks per accumulator group
    static constexpr uint32_t kTmemCols = 512;
    static constexpr size_t kBarOff = (size_t)kStages * kStageBytes + (size_t)kRawStages * kRawBytes;
    static constexpr size_t kSmem = 1024 + kBarOff + 8 * (2 * kStages + 2 * kRawStages + 2 * kAcc + 1) + 16;
};
static_assert(FCfg::kSmem <= 232448, "fit3x shared memory");
static_assert(128 * 129 * 4 <= FCfg::kStages * FCfg::kStageBytes, "fit3x staging tile");

struct FParams {
    char* state;       // layer states, `bytes` apart; M at +64
    size_t bytes;
    int64_t D, n;
    int tiles;         // lower tiles per layer
    unsigned int* err;
};

constexpr int kFitThreads = 320;  // warps 0-3 split, 4-7 epilogue, 8 MMA, 9 TMA
__global__ void __launch_bounds__(kFitThreads, 1) fit3x_kernel(const __grid_constant__ CUtensorMap tm, const FParams p) {
    constexpr int BN = 128;
    using C = FCfg;
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = (uint8_t*)(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
    uint8_t* raw0 = smem + (size_t)C::kStages * C::kStageBytes;
    uint64_t* bars = (uint64_t*)(smem + C::kBarOff);
    uint64_t* full = bars;                          // count 4 (producer warps)
    uint64_t* empty = bars + C::kStages;            // count 1 (MMA commit)
    uint64_t* raw_full = empty + C::kStages;        // count 1 + TMA bytes
    uint64_t* raw_empty = raw_full + C::kRawStages; // count 4 (producer warps)
    uint64_t* acc_full = raw_empty + C::kRawStages; // count 1 (MMA commit): a group is in accumulator a
    uint64_t* acc_empty = acc_full + C::kAcc;       // count 4 (epilogue warps): accumulator a drained
    uint64_t* mma_done = acc_empty + C::kAcc;
    uint32_t* tmem_slot = (uint32_t*)(mma_done + 1);
    volatile int* abort = (volatile int*)(tmem_slot + 1);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    if (threadIdx.x == 0) {
        for (int s = 0; s < C::kStages; ++s) {
            mbar_init(smem_u32(&full[s]), 4);
            mbar_init(smem_u32(&empty[s]), 1);
        }
        for (int r = 0; r < C::kRawStages; ++r) {
            mbar_init(smem_u32(&raw_full[r]), 1);
            mbar_init(smem_u32(&raw_empty[r]), 4);
        }
        for (int a = 0; a < C::kAcc; ++a) {
            mbar_init(smem_u32(&acc_full[a]), 1);
            mbar_init(smem_u32(&acc_empty[a]), 4);
        }
        mbar_init(smem_u32(mma_done), 1);
        *abort = 0;
        fence_mbar_init();
    }
    if (warp == 4) {
        tmem_alloc(smem_u32(tmem_slot), C::kTmemCols);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *tmem_slot;

    const int layer = blockIdx.x / p.tiles;
    const int t = blockIdx.x - layer * p.tiles;
    int by = (int)((sqrtf(8.f * t + 1.f) - 1.f) * 0.5f);  // lower-tile index -> (by, bx), bx <= by
    while ((by + 1) * (by + 2) / 2 <= t) ++by;
    while (by * (by + 1) / 2 > t) --by;
    const int bx = t - by * (by + 1) / 2;
    const bool diag = bx == by;
    const int64_t a0 = (int64_t)by * kBM, b0 = (int64_t)bx * BN;
    const int64_t nkc = (p.n + kKC - 1) / kKC;

    if (warp < 4) {
        // ---------------- split warps: raw chunk (transposed reads) -> hi/lo operand stage
        const int pt = threadIdx.x;
        float4 va[8], vb[8];
        for (int64_t kc = 0; kc < nkc; ++kc) {
            const int r = (int)(kc % C::kRawStages), s = (int)(kc % C::kStages);
            const uint32_t rph = (uint32_t)(kc / C::kRawStages) & 1u, ph = (uint32_t)(kc / C::kStages) & 1u;
            bool got = true;
            if (lane == 0) got = wait_bounded(smem_u32(&raw_full[r]), rph, abort, p.err);
            got = __shfl_sync(0xffffffffu, got, 0);
            __syncwarp();
            if (!got) break;
            const uint8_t* raw = raw0 + (size_t)r * C::kRawBytes;
            load_raw_t(raw, va, pt);
            if (!diag) load_raw_t(raw + C::kABytes, vb, pt);
            __syncwarp();
            if (lane == 0) mbar_arrive(smem_u32(&raw_empty[r]));
            if (lane == 0) got = wait_bounded(smem_u32(&empty[s]), ph ^ 1u, abort, p.err);
            got = __shfl_sync(0xffffffffu, got, 0);
            __syncwarp();
            if (!got) break;
            uint8_t* st = smem + (size_t)s * C::kStageBytes;
            store_split_t<kBM>(va, st, st + C::kABytes, pt);
            if (!diag) store_split_t<BN>(vb, st + 2 * C::kABytes, st + 3 * C::kABytes, pt);
            fence_proxy_async();
            __syncwarp();
            if (lane == 0) mbar_arrive(smem_u32(&full[s]));
        }
    } else if (warp == 9) {
        if (lane == 0) {
            // ---------------- TMA producer: raw chunks of 32 examples, features a0.. (and b0..)
            const int xa = (int)(layer * p.D + a0), xb = (int)(layer * p.D + b0);
            const uint32_t bytes = diag ? C::kABytes : C::kRawBytes;
            uint32_t last_par[C::kRawStages];
            bool issued[C::kRawStages];
            for (int r = 0; r < C::kRawStages; ++r) issued[r] = false;
            for (int64_t kc = 0; kc < nkc; ++kc) {
                const int r = (int)(kc % C::kRawStages);
                const uint32_t rph = (uint32_t)(kc / C::kRawStages) & 1u;
                if (!wait_bounded(smem_u32(&raw_empty[r]), rph ^ 1u, abort, p.err)) break;
                const uint32_t dst = smem_u32(raw0 + (size_t)r * C::kRawBytes), bar = smem_u32(&raw_full[r]);
                const int y = (int)(kc * kKC);
                mbar_arrive_tx(bar, bytes);
#pragma unroll
                for (int b = 0; b < 4; ++b) tma_load_2d(dst + (uint32_t)b * 4096u, &tm, xa + 32 * b, y, bar);
                if (!diag)
#pragma unroll
                    for (int b = 0; b < 4; ++b)
                        tma_load_2d(dst + C::kABytes + (uint32_t)b * 4096u, &tm, xb + 32 * b, y, bar);
                issued[r] = true;
                last_par[r] = rph;
            }
            // copies still in flight when the consumers stopped early land before the CTA exits
            for (int r = 0; r < C::kRawStages; ++r)
                if (issued[r]) {
                    const uint64_t t0 = global_ns();
                    while (!mbar_try_wait(smem_u32(&raw_full[r]), last_par[r]))
                        if (global_ns() - t0 > kTimeoutNs) {
                            atomicOr(p.err, kErrTimeout);
                            break;
                        }
                }
        }
    } else if (warp == 8) {
        if (lane == 0) {
            // ---------------- MMA issuer
            const uint32_t idesc = idesc_tf32(kBM, BN);
            for (int64_t kc = 0; kc < nkc; ++kc) {
                const int s = (int)(kc % C::kStages);
                const uint32_t ph = (uint32_t)(kc / C::kStages) & 1u;
                const int64_t g = kc / C::kGroup;  // group g goes to accumulator g % kAcc, its use g / kAcc
                const int a = (int)(g % C::kAcc);
                const bool start = kc % C::kGroup == 0;
                if (start && g >= C::kAcc &&
                    !wait_bounded(smem_u32(&acc_empty[a]), (uint32_t)((g / C::kAcc) - 1) & 1u, abort, p.err))
                    break;
                if (!wait_bounded(smem_u32(&full[s]), ph, abort, p.err)) break;
                tc_fence_after();
                const uint32_t st = smem_u32(smem + (size_t)s * C::kStageBytes);
                const uint64_t ahi = sw128_desc(st), alo = sw128_desc(st + C::kABytes);
                const uint64_t bhi = diag ? ahi : sw128_desc(st + 2 * C::kABytes);
                const uint64_t blo = diag ? alo : sw128_desc(st + 3 * C::kABytes);
                const uint32_t d = tmem + (uint32_t)a * BN;
#pragma unroll
                for (int k = 0; k < kKC / 8; ++k) {
                    mma_tf32(d, ahi + 2 * k, bhi + 2 * k, idesc, (start && k == 0) ? 0u : 1u);
                    mma_tf32(d, ahi + 2 * k, blo + 2 * k, idesc, 1u);
                    mma_tf32(d, alo + 2 * k, bhi + 2 * k, idesc, 1u);
                }
                mma_commit(smem_u32(&empty[s]));
                if (kc % C::kGroup == C::kGroup - 1 || kc == nkc - 1) mma_commit(smem_u32(&acc_full[a]));
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
        // ---------------- epilogue (warps 4-7): drain each group's accumulator into fp32
        // registers (one row of the tile per thread), then M += the sum
        const int q = warp & 3;
        const int row = q * 32 + lane;
        const uint32_t tbase = tmem + ((uint32_t)(q * 32) << 16);
        const int64_t ngroups = (nkc + C::kGroup - 1) / C::kGroup;
        float acc[BN];
#pragma unroll
        for (int c = 0; c < BN; ++c) acc[c] = 0.f;
        bool ok = true;
        for (int64_t g = 0; g < ngroups; ++g) {
            const int a = (int)(g % C::kAcc);
            bool got = true;
            if (lane == 0) got = wait_bounded(smem_u32(&acc_full[a]), (uint32_t)(g / C::kAcc) & 1u, abort, p.err);
            got = __shfl_sync(0xffffffffu, got, 0);
            if (!got) {
                ok = false;
                break;
            }
            tc_fence_after();
#pragma unroll
            for (int c0 = 0; c0 < BN; c0 += 16) {
                float v[16];
                tmem_ld16(tbase + (uint32_t)(a * BN + c0), v);
#pragma unroll
                for (int i = 0; i < 16; ++i) acc[c0 + i] += v[i];
            }
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(smem_u32(&acc_empty[a]));
        }
        // the tile's sums to shared memory (the operand stages are free once the last group
        // has landed: every stage was consumed by its MMAs), row stride 129: conflict-free
        if (ok) {
            float* stg = (float*)smem;
#pragma unroll
            for (int c = 0; c < BN; ++c) stg[row * (BN + 1) + c] = acc[c];
        }
    }
    tc_fence_before();
    __syncthreads();
    if (!*abort) {
        // M += tile, coalesced: warp w takes rows 4j..4j+3 for j = w, w + 10, ..., lane the
        // columns lane + 32i; all 16 old values of a batch are loaded before any store
        const float* stg = (const float*)smem;
        float* M = (float*)(p.state + (size_t)layer * p.bytes + 64);
        for (int j = warp; j < kBM / 4; j += kFitThreads / 32) {
            float old[4][BN / 32];
#pragma unroll
            for (int r = 0; r < 4; ++r)
#pragma unroll
                for (int i = 0; i < BN / 32; ++i) {
                    const int64_t a = a0 + 4 * j + r, b = b0 + lane + 32 * i;
                    old[r][i] = (a < p.D && b < p.D) ? M[a * p.D + b] : 0.f;
                }
#pragma unroll
            for (int r = 0; r < 4; ++r)
#pragma unroll
                for (int i = 0; i < BN / 32; ++i) {
                    const int64_t a = a0 + 4 * j + r, b = b0 + lane + 32 * i;
                    if (a < p.D && b < p.D) M[a * p.D + b] = old[r][i] + stg[(4 * j + r) * (BN + 1) + lane + 32 * i];
                }
        }
    }
    if (warp == 4) {
        tc_fence_after();
        tmem_dealloc(tmem, C::kTmemCols);
    }
}

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

// 2-D map over fp32 X[rows][ld] (features 0..K-1 used): box 32 features x box_rows rows,
// 128-byte swizzle, zero fill past K and past the last row.
bool make_map_f32(CUtensorMap* tm, const float* X, int64_t rows, int64_t K, int64_t ld, int box_rows) {
    EncodeTiledFn enc = encode_fn();
    if (!enc) return false;
    cuuint64_t dims[2] = {(cuuint64_t)K, (cuuint64_t)rows};
    cuuint64_t strides[1] = {(cuuint64_t)(ld * 4)};
    cuuint32_t box[2] = {(cuuint32_t)kKC, (cuuint32_t)box_rows};
    cuuint32_t estr[2] = {1, 1};
    return enc(tm, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 2, const_cast<float*>(X), dims, strides, box, estr,
               CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
               CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// 3-D map over nz batch entries of fp32 X[rows][ld] (features 0..K-1 used), entry z at byte
// offset z * z_bytes from X; box 32 features x box_rows rows x 1 entry, 128-byte swizzle.
bool make_map_f32_3d(CUtensorMap* tm, const float* X, int64_t rows, int64_t K, int64_t ld, int64_t nz,
                     size_t z_bytes, int box_rows) {
    EncodeTiledFn enc = encode_fn();
    if (!enc) return false;
    cuuint64_t dims[3] = {(cuuint64_t)K, (cuuint64_t)rows, (cuuint64_t)nz};
    cuuint64_t strides[2] = {(cuuint64_t)(ld * 4), (cuuint64_t)z_bytes};
    cuuint32_t box[3] = {(cuuint32_t)kKC, (cuuint32_t)box_rows, 1};
    cuuint32_t estr[3] = {1, 1, 1};
    return enc(tm, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 3, const_cast<float*>(X), dims, strides, box, estr,
               CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
               CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

template <int BN>
cudaError_t launch_bn(GParams p, cudaStream_t s, int64_t nz = 1, size_t a_z_bytes = 0, size_t b_z_bytes = 0) {
    using C = GCfg<BN>;
    CUtensorMap tmA, tmB;
    if (nz > 1) {
        if (!make_map_f32_3d(&tmA, p.A, p.n_t, p.K, p.lda, nz, a_z_bytes, kBM) ||
            !make_map_f32_3d(&tmB, p.B, p.n_q, p.K, p.ldb, nz, b_z_bytes, BN))
            return cudaErrorInvalidValue;
        p.batched = 1;
    } else if (!make_map_f32(&tmA, p.A, p.n_t, p.K, p.lda, kBM) || !make_map_f32(&tmB, p.B, p.n_q, p.K, p.ldb, BN)) {
        return cudaErrorInvalidValue;
    }
    static int sms = 0;
    if (!sms) {
        int dev = 0;
        cudaGetDevice(&dev);
        cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
        if (sms <= 0) sms = 1;
    }
    const int64_t tiles_m = (p.n_t + kBM - 1) / kBM, tiles_n = (p.n_q + BN - 1) / BN;
    const int64_t tiles = p.lower ? tiles_n * (tiles_n + 1) / 2 : tiles_m * tiles_n;
    const int64_t nkc = ((p.kslice ? p.kslice : p.K) + kKC - 1) / kKC;
    int cs = 1;
    // split K over a cluster only while the tiles of all batch entries leave SMs idle
    while (cs < 4 && tiles * p.splits * nz * cs * 2 <= sms && nkc >= 8 * cs * 2) cs *= 2;
    // the leader's stage buffers must hold the members' partial tiles
    while (cs > 1 && (size_t)(cs - 1) * kBM * BN * 4 > (size_t)C::kStages * C::kStageBytes) cs >>= 1;
    p.cs = cs;
    p.tiles_n = (int)tiles_n;
    if (cs == 1 && p.splits == 1 && !p.kslice && nkc <= 64 && tiles * nz > sms) {
        // more tiles than SMs with short K: one persistent CTA per SM walks the tiles
        using P = PCfg<BN>;
        p.tiles_z = tiles;
        p.nz = (int)nz;
        cudaError_t e = smem_attr_once<gemm3x_persist_kernel<BN>>((int)P::kSmem);
        if (e != cudaSuccess) return e;
        note_launches(1);
        gemm3x_persist_kernel<BN><<<(unsigned)sms, kThreadsP, P::kSmem, s>>>(tmA, tmB, p);
        return cudaGetLastError();
    }
    cudaError_t e = smem_attr_once<score3x_kernel<BN>>((int)C::kSmem);
    if (e != cudaSuccess) return e;
    cudaLaunchConfig_t cfg = {};
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = (unsigned)cs;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    cfg.gridDim = dim3((unsigned)(tiles * cs), (unsigned)p.splits, (unsigned)nz);
    cfg.blockDim = dim3(kThreads);
    cfg.dynamicSmemBytes = C::kSmem;
    cfg.stream = s;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    note_launches(1);
    e = cudaLaunchKernelEx(&cfg, score3x_kernel<BN>, tmA, tmB, p);
    if (e != cudaSuccess) return e;
    return cudaGetLastError();
}

}  // namespace

bool score_tc_supported(tda_dtype qdt, const void* Qhat, int64_t n_q, int64_t ld_q, const float* Phi, int64_t n_t,
                        int64_t ld_phi, int64_t D) {
    static int sm103 = -1;
    if (sm103 < 0) {
        int dev = 0, major = 0, minor = 0;
        cudaGetDevice(&dev);
        cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev);
        cudaDeviceGetAttribute(&minor, cudaDevAttrComputeCapabilityMinor, dev);
        sm103 = (major == 10 && minor == 3) ? 1 : 0;
    }
    if (!sm103 || qdt != TDA_F32 || !encode_fn()) return false;
    // TMA: 32-bit coordinates, row strides of whole 16-byte groups below 2^40 bytes
    if (n_q < 1 || n_t < 1 || D < 64 || D >= (1LL << 31) || n_q > (1LL << 24) || n_t > (1LL << 31) / kBM * kBM)
        return false;
    if (ld_q * 4 >= (1LL << 40) || ld_phi * 4 >= (1LL << 40)) return false;
    if ((ld_q & 3) || (ld_phi & 3)) return false;
    if (((uintptr_t)Qhat & 15) || ((uintptr_t)Phi & 15)) return false;
    return true;
}

cudaError_t launch_score_tc(const float* Qhat, int64_t n_q, int64_t ld_q, const float* Phi, int64_t n_t, int64_t ld_phi,
                            int64_t D, float* S, int64_t ld_S, float beta, unsigned int* err, cudaStream_t s) {
    GParams p{};
    p.A = Phi;
    p.B = Qhat;
    p.S = S;
    p.n_t = n_t;
    p.n_q = n_q;
    p.K = D;
    p.lda = ld_phi;
    p.ldb = ld_q;
    p.ld_S = ld_S;
    p.beta = beta;
    p.alpha = 1.f;
    p.kslice = 0;
    p.slab = 0;
    p.splits = 1;
    p.err = err;
    if (n_q <= 64) return launch_bn<64>(p, s);
    return launch_bn<128>(p, s);
}

int score_tc_tiles(int64_t n_q, int64_t n_t) {
    const int64_t bn = n_q <= 64 ? 64 : 128;
    const int64_t t = ((n_t + kBM - 1) / kBM) * ((n_q + bn - 1) / bn);
    return t > (1 << 30) ? (1 << 30) : (int)t;
}

// Partial scores of `splits` feature slices: part[z][q][i] = sum over slice z of
// Phi[i][f] Qhat[q][f] (slices of a multiple of 32 features; part holds
// splits * n_q * n_t floats). The caller sums the slabs.
cudaError_t launch_score_tc_slices(const float* Qhat, int64_t n_q, int64_t ld_q, const float* Phi, int64_t n_t,
                                   int64_t ld_phi, int64_t D, int splits, float* part, unsigned int* err,
                                   cudaStream_t s) {
    GParams p{};
    p.A = Phi;
    p.B = Qhat;
    p.n_t = n_t;
    p.n_q = n_q;
    p.K = D;
    p.lda = ld_phi;
    p.ldb = ld_q;
    int64_t kslice = (D + splits - 1) / splits;
    kslice = (kslice + kKC - 1) / kKC * kKC;
    p.kslice = kslice;
    p.splits = (int)((D + kslice - 1) / kslice);
    p.slab = n_q * n_t;
    p.S = part;
    p.ld_S = n_t;
    p.beta = 0.f;
    p.alpha = 1.f;
    p.err = err;
    if (p.splits > 65535) return cudaErrorInvalidValue;
    if (n_q <= 64) return launch_bn<64>(p, s);
    return launch_bn<128>(p, s);
}

cudaError_t launch_gemm_nt_tc_batched(const float* A, int64_t n_a, int64_t lda, size_t a_z_bytes, const float* B,
                                      int64_t n_b, int64_t ldb, size_t b_z_bytes, int64_t K, float* C, int64_t ldc,
                                      int64_t c_z, int64_t nz, float alpha, float beta, bool lower,
                                      unsigned int* err, cudaStream_t s);

// C[n][m] = beta * C[n][m] + alpha * sum_k A[m][k] B[n][k] (C row stride ldc): the
// score GEMM with a sign, used by the blocked Cholesky and triangular solves. With
// lower = true, A and B must be the same n x n operand rows (a symmetric rank-K
// update) and only the 128 x 128 tiles on or below the diagonal (m0 <= n0) are
// formed; entries above the diagonal inside a diagonal tile are written too.
cudaError_t launch_gemm_nt_tc(const float* A, int64_t n_a, int64_t lda, const float* B, int64_t n_b, int64_t ldb,
                              int64_t K, float* C, int64_t ldc, float alpha, float beta, bool lower,
                              unsigned int* err, cudaStream_t s) {
    return launch_gemm_nt_tc_batched(A, n_a, lda, 0, B, n_b, ldb, 0, K, C, ldc, 0, 1, alpha, beta, lower, err, s);
}

cudaError_t launch_gemm_nt_tc_batched(const float* A, int64_t n_a, int64_t lda, size_t a_z_bytes, const float* B,
                                      int64_t n_b, int64_t ldb, size_t b_z_bytes, int64_t K, float* C, int64_t ldc,
                                      int64_t c_z, int64_t nz, float alpha, float beta, bool lower,
                                      unsigned int* err, cudaStream_t s) {
    if (nz < 1 || nz > 65535) return cudaErrorInvalidValue;
    if (nz > 1 && ((a_z_bytes & 15) || (b_z_bytes & 15) || !a_z_bytes || !b_z_bytes)) return cudaErrorInvalidValue;
    GParams p{};
    p.A = A;
    p.B = B;
    p.S = C;
    p.n_t = n_a;
    p.n_q = n_b;
    p.K = K;
    p.lda = lda;
    p.ldb = ldb;
    p.ld_S = ldc;
    p.beta = beta;
    p.alpha = alpha;
    p.lower = lower ? 1 : 0;
    p.kslice = 0;
    p.slab = 0;
    p.splits = 1;
    p.s_z = c_z;
    p.err = err;
    if (lower && (n_a != n_b || n_b <= 64)) return cudaErrorInvalidValue;
    if (n_b <= 64) return launch_bn<64>(p, s, nz, a_z_bytes, b_z_bytes);
    return launch_bn<128>(p, s, nz, a_z_bytes, b_z_bytes);
}

bool gemm_tc_available() {
    static int ok = -1;
    if (ok < 0) {
        int dev = 0, major = 0, minor = 0;
        cudaGetDevice(&dev);
        cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev);
        cudaDeviceGetAttribute(&minor, cudaDevAttrComputeCapabilityMinor, dev);
        ok = (major == 10 && minor == 3 && encode_fn()) ? 1 : 0;
    }
    return ok == 1;
}

bool fit_tc_supported(int n_layers, int64_t D, const float* phi, int64_t n, int64_t ld) {
    int dev = 0, major = 0, minor = 0;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev);
    cudaDeviceGetAttribute(&minor, cudaDevAttrComputeCapabilityMinor, dev);
    if (!(major == 10 && minor == 3) || !encode_fn()) return false;
    // TMA: 32-bit coordinates, 16-byte aligned base and row stride below 2^40 bytes, feature
    // coordinates a multiple of 4 (every tile starts at l*D + 128*j)
    if (D < 128 || (D & 3) || (ld & 3) || ((uintptr_t)phi & 15)) return false;
    if ((int64_t)n_layers * D >= (1LL << 31) || n >= (1LL << 31) - kKC || ld * 4 >= (1LL << 40)) return false;
    return true;
}

cudaError_t launch_fit_tc(int n_layers, int64_t D, void* state, size_t state_bytes, const float* phi, int64_t n,
                          int64_t ld, unsigned int* err, cudaStream_t s) {
    using C = FCfg;
    const int64_t nt = (D + kBM - 1) / kBM;
    // features of all layers, examples as rows; zero fill past the last layer's features and the last example
    CUtensorMap tm;
    if (!make_map_f32(&tm, phi, n, (int64_t)n_layers * D, ld, kKC)) return cudaErrorInvalidValue;
    FParams p{};
    p.state = (char*)state;
    p.bytes = state_bytes;
    p.D = D;
    p.n = n;
    p.tiles = (int)(nt * (nt + 1) / 2);
    p.err = err;
    cudaError_t e = smem_attr_once<fit3x_kernel>((int)C::kSmem);
    if (e != cudaSuccess) return e;
    note_launches(1);
    fit3x_kernel<<<(unsigned)(p.tiles * n_layers), kFitThreads, C::kSmem, s>>>(tm, p);
    return cudaGetLastError();
}

}  // namespace tda
