// k_project_tc.cu -- factored projection (Eq. 2) on the 5th-generation tensor
// cores of sm_103a: tcgen05.mma with TMEM accumulators, operands staged in
// shared memory by TMA (factors) and by generator warps (signs).
//
// For every 128-row token tile:
//   At = A_tile S_in   (128 x k_in,  K = d_in)    tcgen05, accumulators in TMEM
//   Bt = B_tile S_out  (128 x k_out, K = d_out)   tcgen05, accumulators in TMEM
//   Phi_n += Bt^T At   (k_out x k_in, over the tile's tokens of example n) on
//                      CUDA cores, fp32
// and finally Phi_n *= 1/sqrt(k_in k_out). The signs S (App. A.2) come from the
// counter hash: one 64-bit word gives the 64 signs of one column over one
// 64-row K chunk, which is one 128-byte row of the K-major, 128B-swizzled
// operand tile, so the projection matrices never touch global memory.
//
// Token tiles: for T > 64 a tile is 128 consecutive tokens of one example (the
// last one zero-filled past T); for T <= 64 a tile packs floor(128 / T) whole
// examples (the factors of consecutive examples are consecutive rows), so short
// sequences do not leave most of each MMA empty.
//
// A pipeline stage holds G token tiles (G = 2 for large batches) that share
// one sign tile: the signs of a K chunk do not depend on the tokens, so
// generating them once for G tiles halves the generators' work and the MMA
// commits per byte streamed.
//
// The kernel streams every factor byte once from HBM; its arithmetic
// intensity (~k flop/B, k <= 128) is below the tensor-core ridge, so it is
// HBM-bound and the pipeline is sized for bytes in flight.
//
// k = 128 (K = 128): At | Bt of one tile fill 256 TMEM columns, so the two
// accumulator buffers take all 512 and a stage holds one token tile. With the
// optional workspace both sides' sign tables are written once per call and
// brought in by TMA beside the factor tiles instead of by the generator warps.
//
// Staging: the epilogue stages a tile's fp32 rows in shared memory in parts of
// SR token rows (32 where every CTA owns whole examples or balanced ranges, 64
// or 128 otherwise); fewer staged rows leave room for more stages in the ring.
//
// Work split: whole examples per CTA (example slots cid, cid + ncl, ...);
// below one example per SM a cluster of 2 or 4 CTAs shares an example's token
// tiles and reduces the partial K x K blocks over distributed shared memory;
// with the workspace (balanced ranges) every CTA takes an equal contiguous run
// of token tiles and an example split between CTAs is summed from partial
// blocks, in CTA order, by the last of them to finish (store_phi_bal).
//
// Warp roles (256 threads, one persistent CTA per SM):
//   warp 0  TMA producer: 128x64 bf16 factor tiles into the stage ring
//   warp 1  TMEM allocator; lane 0 issues the MMAs
//   warps 2-3  sign generators: k x 64 bf16 +-1 tiles into the stage ring,
//           each warp one half of every 128-byte row
//   warps 4-7  epilogue: TMEM -> registers -> shared -> token contraction
// Accumulators are double-buffered in TMEM, so the epilogue of one group of
// tiles overlaps the MMAs of the next. Every wait is bounded (about 1 s); on
// expiry the kernel records kErrTimeout in the device error word, drains its
// copies, frees its TMEM and returns.
#include <cuda.h>
#include <cuda_bf16.h>

#include <cstring>
#include <mutex>
#include <type_traits>

#include "tda_internal.cuh"

namespace tda {
namespace {

constexpr int kThreads = 256;
constexpr int kTileM = 128;            // tokens per tile (MMA M)
constexpr int kChunkK = 64;            // K elements per stage (128 bytes of bf16)
constexpr uint32_t kTileBytes = kTileM * kChunkK * 2;  // 16 KiB per factor tile
constexpr size_t kSmemMax = 232448;    // 227 KiB of dynamic shared memory per CTA
constexpr int kMaxStages = 12;

// SR: token rows the epilogue stages in shared memory at a time (32, 64 or 128).
// Fewer rows leave room for more stages in the ring, i.e. more factor bytes in
// flight per SM, which is what an HBM-bound stream needs; a whole tile (128)
// is staged where the epilogue needs every row at once (packed short
// sequences, the K-FAC covariances, the factor output).
// LUT: shared memory for the sign-expansion table (K = 128 with generator warps;
// sign tiles that arrive by TMA need none, which leaves room for one more stage).
template <int K, int G, int SR = (K > 64 ? kTileM / 2 : kTileM), bool LUT = (K > 64)>
struct Cfg {
    static constexpr int kK = K;
    static constexpr uint32_t kSignBytes = K * 128;                       // K rows x 128 bytes
    static constexpr uint32_t kStageBytes = G * kTileBytes + kSignBytes;  // G factor tiles, then signs
    static constexpr int kStageLd = K + 4;                                // padded fp32 staging row
    // K = 128: signs are expanded through a byte table, two columns per generator lane
    static constexpr bool kHalf = K > 64;
    // the epilogue stages and contracts a tile's token rows in parts of SR rows
    static constexpr bool kParted = SR < kTileM;
    static constexpr int kStageRows = SR;
    static_assert(SR == 32 || SR == 64 || SR == 128, "whole TMEM lane quadrants per part");
    static constexpr int kAccCols = 2 * K;                                // At | Bt of one tile
    static constexpr int kBufCols = G * kAccCols;                         // one accumulator buffer
    // tcgen05.alloc takes a power of two from 32 to 512 columns
    static constexpr uint32_t kTmemCols = 2 * kBufCols <= 32    ? 32
                                          : 2 * kBufCols <= 64  ? 64
                                          : 2 * kBufCols <= 128 ? 128
                                          : 2 * kBufCols <= 256 ? 256
                                                                : 512;
    static constexpr size_t kSmemStage = 2ull * kStageRows * kStageLd * 4;
    // a cluster of cs CTAs reduces cs - 1 partial K x K blocks inside the leader's staging rows
    static constexpr int kMaxCs = (int)(2 * kStageRows * kStageLd / (K * K)) + 1;
    static constexpr size_t kSmemBarsMax = 8 * (3 * kMaxStages + 7) + 16;
    // K = 128: a 256-entry table expands a byte of sign bits into eight bf16 signs
    static constexpr bool kLut = LUT;
    static constexpr size_t kLutBytes = kLut ? 256 * 16 : 0;
    static constexpr size_t kLutMax = kLut ? kLutBytes + 8 : 0;
    static constexpr int kFit = (int)((kSmemMax - 1024 - kSmemStage - kSmemBarsMax - kLutMax) / kStageBytes);
    static constexpr int kStages = kFit > kMaxStages ? kMaxStages : kFit;
    static constexpr size_t kSmemBars = 8 * (3 * kStages + 7) + 16;
    static constexpr size_t kBarsOff = (size_t)kStages * kStageBytes + kSmemStage;  // after ring and staging
    static constexpr size_t kLutOff = (kBarsOff + kSmemBars + 15) / 16 * 16;
    static constexpr size_t kSmem = 1024 + (kLut ? kLutOff + kLutBytes : kBarsOff + kSmemBars);
    // contraction blocking: 16 row groups x 8 column groups of threads
    static constexpr int RB = K / 16 > 0 ? K / 16 : 1;
    static constexpr int CB = K / 8;
    static_assert(kStages >= 3 && kSmem <= kSmemMax, "shared memory per CTA");
    static_assert(!kHalf || G == 1, "K = 128 fills TMEM with one double-buffered tile");
    static_assert(!kHalf || kParted, "K = 128 stages at most half a tile");
    static_assert(!kHalf || (kThreads == 256 && K == 128), "one thread per sign-table entry; two columns per lane");
    static_assert(kStageBytes % 1024 == 0 && 2 * kBufCols <= (int)kTmemCols && kTmemCols <= 512,
                  "operand alignment / TMEM columns");
};

struct Params {
    int64_t N, T, d_in, d_out, ld_phi;
    int64_t n_slots;  // example slots: examples (pack == 1) or groups of `pack` examples
    uint64_t key_in, key_out;
    float scale;
    float* phi;
    unsigned int* err;
    int n_ttiles;     // token tiles per slot
    int pack;         // examples per token tile (T <= 64), else 1
    int nk_in, nk_out;
    int cs;           // CTAs per cluster sharing one example's token tiles (1, 2 or 4)
    float* cov;       // K-FAC: per-CTA partial sums of At^T At and Bt^T Bt ([grid][2][K*K])
    float* fout;      // factor output: At rows [N*T][K], then Bt rows [N*T][K] (unscaled signs)
    // balanced ranges (BAL): CTA c owns token tiles [n_units*c/grid, n_units*(c+1)/grid) of the
    // flattened (example, tile) sequence; an example split across CTAs leaves an unscaled partial
    // block per CTA in part ([grid][2][K*K]: slot 0 = the CTA's first example, 1 = its last) and
    // the last of them to finish (counter cnt[first CTA of the example]) sums them in CTA order
    int64_t n_units;
    float* part;
    unsigned int* cnt;
};

#include "tc_ptx.cuh"

// The sequence of token tiles ("units") one CTA works on, identical for every
// warp role: example slots cid, cid + ncl, ... and, within a slot, the token
// tiles crank, crank + cs, ...
struct Units {
    int64_t x;
    int tt;
    __device__ __forceinline__ void first(const Params&, uint32_t cid, uint32_t crank) {
        x = cid;
        tt = (int)crank;
    }
    // Next group of up to G units into gx/gt; returns how many (0 = finished).
    template <int G>
    __device__ __forceinline__ int take(const Params& p, uint32_t ncl, uint32_t crank, int64_t* gx, int* gt) {
        int n = 0;
#pragma unroll
        for (int u = 0; u < G; ++u)
            if (x < p.n_slots) {
                gx[u] = x;
                gt[u] = tt;
                ++n;
                tt += p.cs;
                if (tt >= p.n_ttiles) {
                    tt = (int)crank;
                    x += ncl;
                }
            }
        return n;
    }
};

// Balanced ranges: the same contiguous run of token tiles for every warp role.
struct TileRange {
    int64_t t, t1;
    __device__ __forceinline__ void first(const Params& p, uint32_t, uint32_t) {
        t = p.n_units * (int64_t)blockIdx.x / gridDim.x;
        t1 = p.n_units * ((int64_t)blockIdx.x + 1) / gridDim.x;
    }
    template <int G>
    __device__ __forceinline__ int take(const Params& p, uint32_t, uint32_t, int64_t* gx, int* gt) {
        int n = 0;
#pragma unroll
        for (int u = 0; u < G; ++u)
            if (t < t1) {
                gx[u] = t / p.n_ttiles;
                gt[u] = (int)(t - gx[u] * p.n_ttiles);
                ++t;
                ++n;
            }
        return n;
    }
};

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

// Phi of example n (K x K partial sums in acc, thread et holding rows
// rg*RB.. and columns cg*CB..) is complete in every CTA of the cluster: reduce
// the members' blocks into the leader (rank 0) over distributed shared memory
// and write it, scaled. The leader's staging rows (free between tiles) receive
// member r's block at offset (r-1)*K*K floats, thread-major.
template <class C>
__device__ __forceinline__ bool store_phi(float (&acc)[C::RB][C::CB], int64_t n, const Params& p, uint32_t crank,
                                          float* stage, uint64_t* red_go, uint64_t* red_full, uint32_t& red_use,
                                          volatile int* abort, int et, int lane) {
    constexpr int K = C::kK;
    const int rg = et >> 3, cg = et & 7;
    if (p.cs > 1) {
        constexpr int kPer = C::RB * C::CB;
        const uint32_t slot = smem_u32(stage) + (uint32_t)(et * kPer) * 4u;
        bool got = true;
        if (crank == 0) {
            if (et == 0)
                for (int r = 1; r < p.cs; ++r) mbar_arrive_remote(smem_u32(red_go), (uint32_t)r);
            if (lane == 0) got = wait_bounded_cluster(smem_u32(red_full), red_use & 1u, abort, p.err);
            got = __shfl_sync(0xffffffffu, got, 0);
            if (epi_any(!got)) return false;
            for (int r = 1; r < p.cs; ++r) {
                const float* part = stage + (r - 1) * K * K + et * kPer;
#pragma unroll
                for (int a = 0; a < C::RB; ++a)
#pragma unroll
                    for (int c = 0; c < C::CB; ++c) acc[a][c] += part[a * C::CB + c];
            }
            epi_sync();  // partials consumed; staging free for the next tile
        } else {
            if (lane == 0) got = wait_bounded_cluster(smem_u32(red_go), red_use & 1u, abort, p.err);
            got = __shfl_sync(0xffffffffu, got, 0);
            if (epi_any(!got)) return false;
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
        if (crank != 0) return true;
    }
    float* out = p.phi + n * p.ld_phi;
#pragma unroll
    for (int a = 0; a < C::RB; ++a)
#pragma unroll
        for (int c = 0; c < C::CB; ++c) out[(rg * C::RB + a) * K + cg * C::CB + c] = acc[a][c] * p.scale;
    return true;
}

// Balanced ranges: Phi of example n (K x K partial sums in acc, layout as in
// store_phi) after this CTA's last tile of it. An example wholly inside the
// CTA's range is written directly; otherwise the partial goes to the CTA's
// slot in p.part, and the last of the example's CTAs to arrive at its counter
// adds all partials in CTA order (the same sum whichever CTA finishes last),
// scales, writes Phi and clears the counter. Nothing waits on another CTA.
template <class C>
__device__ __forceinline__ void store_phi_bal(float (&acc)[C::RB][C::CB], int64_t n, const Params& p, int et,
                                              volatile int* flag) {
    constexpr int K = C::kK;
    const int rg = et >> 3, cg = et & 7;
    const int64_t nt = p.n_ttiles, U = p.n_units, g = gridDim.x, c = blockIdx.x;
    const int64_t u0 = n * nt, u1 = u0 + nt;               // the example's tiles
    const int64_t r0 = U * c / g, r1 = U * (c + 1) / g;     // this CTA's tiles
    float* out = p.phi + n * p.ld_phi;
    if (u0 >= r0 && u1 <= r1) {
#pragma unroll
        for (int a = 0; a < C::RB; ++a)
#pragma unroll
            for (int b = 0; b < C::CB; ++b) out[(rg * C::RB + a) * K + cg * C::CB + b] = acc[a][b] * p.scale;
        return;
    }
    float* mine = p.part + ((size_t)c * 2 + (n == r0 / nt ? 0 : 1)) * K * K;
#pragma unroll
    for (int a = 0; a < C::RB; ++a)
#pragma unroll
        for (int b = 0; b < C::CB; ++b) mine[(rg * C::RB + a) * K + cg * C::CB + b] = acc[a][b];
    __threadfence();
    epi_sync();
    // CTAs holding the example's first and last tiles (every CTA's range is non-empty)
    const int64_t cf = ((u0 + 1) * g - 1) / U, cl = (u1 * g - 1) / U;
    if (et == 0) {
        const unsigned int prev = atomicAdd(p.cnt + cf, 1u);
        const bool last = prev == (unsigned int)(cl - cf);
        if (last) p.cnt[cf] = 0u;  // ready for the next call
        *flag = last ? 1 : 0;
    }
    epi_sync();
    const bool last = *flag != 0;
    epi_sync();  // every thread has read the flag before the next example may set it
    if (!last) return;
    __threadfence();
    float sum[C::RB][C::CB];
#pragma unroll
    for (int a = 0; a < C::RB; ++a)
#pragma unroll
        for (int b = 0; b < C::CB; ++b) sum[a][b] = 0.f;
    for (int64_t c2 = cf; c2 <= cl; ++c2) {
        const int64_t first_ex = (U * c2 / g) / nt;
        const float* part = p.part + ((size_t)c2 * 2 + (n == first_ex ? 0 : 1)) * K * K;
#pragma unroll
        for (int a = 0; a < C::RB; ++a)
#pragma unroll
            for (int b = 0; b < C::CB; ++b) sum[a][b] += __ldcg(part + (rg * C::RB + a) * K + cg * C::CB + b);
    }
#pragma unroll
    for (int a = 0; a < C::RB; ++a)
#pragma unroll
        for (int b = 0; b < C::CB; ++b) out[(rg * C::RB + a) * K + cg * C::CB + b] = sum[a][b] * p.scale;
}

__device__ __forceinline__ uint4 lds128(uint32_t a) {
    uint4 v;
    asm volatile("ld.shared.v4.u32 {%0, %1, %2, %3}, [%4];" : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w) : "r"(a));
    return v;
}

// Entry e of the sign expansion table: bit j of e as the bf16 sign of element j
// (+1 = 0x3F80, -1 = 0xBF80), the layout write_sign_half produces.
__device__ __forceinline__ void init_sign_lut(uint8_t* lut, uint32_t e) {
    uint32_t q[4];
#pragma unroll
    for (int p = 0; p < 4; ++p)
        q[p] = (0x3F80u | (((e >> (2 * p)) & 1u) << 15)) | ((0x3F80u | (((e >> (2 * p + 1)) & 1u) << 15)) << 16);
    *reinterpret_cast<uint4*>(lut + e * 16) = make_uint4(q[0], q[1], q[2], q[3]);
}

// The eight 16-byte chunks of one sign-tile row (the 64 signs of sign word w)
// from the expansion table at shared address lut: one table read per byte.
__device__ __forceinline__ void expand_signs(uint4 (&q)[8], uint64_t w, uint32_t lut) {
#pragma unroll
    for (int c = 0; c < 8; ++c) q[c] = lds128(lut + ((((uint32_t)(w >> (8 * c))) & 0xFFu) << 4));
}

// Row n of a K-major 128B-swizzled sign tile from its eight expanded chunks.
__device__ __forceinline__ void store_sign_row(uint8_t* tile, int n, const uint4 (&q)[8]) {
    uint8_t* row = tile + (n >> 3) * 1024 + (n & 7) * 128;
#pragma unroll
    for (int c = 0; c < 8; ++c) *reinterpret_cast<uint4*>(row + ((c ^ (n & 7)) << 4)) = q[c];
}

// KF: also accumulate the K-FAC factor covariances. FO: write the projected
// factors At, Bt of every token instead of contracting them into Phi. SL: the
// sign tiles come by TMA from a precomputed table (tmSA, tmSB: [K][d] bf16, a
// side's S transposed) instead of the generator warps.
template <int K, int G, bool KF, bool FO, bool SL = false, int SR = Cfg<K, G>::kStageRows, bool BAL = false>
__global__ void __launch_bounds__(kThreads, 1)
project_tc_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
                  const __grid_constant__ CUtensorMap tmSA, const __grid_constant__ CUtensorMap tmSB,
                  const Params p) {
    using C = Cfg<K, G, SR, (K > 64) && !SL>;
    static_assert(!C::kParted || (!KF && !FO), "the K-FAC and factor-output epilogues stage whole tiles");
    static_assert(!BAL || C::kParted, "balanced ranges use the parted epilogue");
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = (uint8_t*)(((uintptr_t)smem_raw + 1023) & ~(uintptr_t)1023);
    uint8_t* sA = smem;                           // kStages x [G factor tiles | sign tile]
    float* stX = (float*)(sA + (size_t)C::kStages * C::kStageBytes);  // [128 or 64][K+4] At rows
    float* stY = stX + C::kStageRows * C::kStageLd;  // [128 or 64][K+4] Bt rows
    uint64_t* bars = (uint64_t*)(smem + C::kBarsOff);
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
    if constexpr (C::kLut) init_sign_lut(smem + C::kLutOff, threadIdx.x);  // kThreads == 256 entries
    if (warp == 1) {
        tmem_alloc(smem_u32(tmem_slot), C::kTmemCols);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    cluster_sync();  // every CTA's barriers exist before any remote arrive
    tc_fence_after();
    const uint32_t tmem = *tmem_slot;
    const uint32_t crank = cluster_rank(), cid = blockIdx.x / p.cs, ncl = gridDim.x / p.cs;
    const int nk_tot = p.nk_in + p.nk_out;
    int64_t gx[G];
    int gt[G];
    typename std::conditional<BAL, TileRange, Units>::type it;
    it.first(p, cid, crank);

    if (warp == 0 && lane == 0) {
        // ---------------- TMA producer
        uint32_t last_par[kMaxStages];
        bool issued[kMaxStages];
        for (int s = 0; s < C::kStages; ++s) issued[s] = false;
        uint32_t ring = 0;
        bool ok = true;
        for (int ng; ok && (ng = it.take<G>(p, ncl, crank, gx, gt)) > 0;)
            for (int kc = 0; kc < nk_tot; ++kc, ++ring) {
                const int s = ring % C::kStages;
                const uint32_t ph = (ring / C::kStages) & 1u;
                if (!wait_bounded(smem_u32(&empty[s]), ph ^ 1u, abort, p.err)) {
                    ok = false;
                    break;
                }
                const bool side_b = kc >= p.nk_in;
                const int d0 = (side_b ? kc - p.nk_in : kc) * kChunkK;
                mbar_arrive_tx(smem_u32(&full[s]), (uint32_t)ng * kTileBytes + (SL ? C::kSignBytes : 0u));
                if constexpr (SL)
                    tma_load_3d(smem_u32(sA + (size_t)s * C::kStageBytes + (size_t)G * kTileBytes),
                                side_b ? &tmSB : &tmSA, d0, 0, 0, smem_u32(&full[s]));
                for (int u = 0; u < ng; ++u) {
                    // packed tiles: row x * pack * T of the [N*T][d] view; else tile tt of example x
                    const int row = p.pack > 1 ? (int)(gx[u] * p.pack * p.T) : gt[u] * kTileM;
                    const int ex = p.pack > 1 ? 0 : (int)gx[u];
                    tma_load_3d(smem_u32(sA + (size_t)s * C::kStageBytes + (size_t)u * kTileBytes),
                                side_b ? &tmB : &tmA, d0, row, ex, smem_u32(&full[s]));
                }
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
        uint32_t ring = 0, grp = 0;
        bool ok = true;
        const uint32_t idesc = idesc_bf16(kTileM, K);
        for (int ng; ok && (ng = it.take<G>(p, ncl, crank, gx, gt)) > 0; ++grp) {
            const uint32_t b = grp & 1u, use = grp >> 1;
            if (!wait_bounded(smem_u32(&tempty[b]), (use & 1u) ^ 1u, abort, p.err)) {
                ok = false;
                break;
            }
            tc_fence_after();
            for (int kc = 0; kc < nk_tot; ++kc, ++ring) {
                const int s = ring % C::kStages;
                const uint32_t ph = (ring / C::kStages) & 1u;
                if (!wait_bounded(smem_u32(&full[s]), ph, abort, p.err) ||
                    (!SL && !wait_bounded(smem_u32(&sready[s]), ph, abort, p.err))) {
                    ok = false;
                    break;
                }
                tc_fence_after();
                const bool side_b = kc >= p.nk_in;
                const int kk = side_b ? kc - p.nk_in : kc;
                uint8_t* stage = sA + (size_t)s * C::kStageBytes;
                const uint64_t bd = sw128_desc(smem_u32(stage + (size_t)G * kTileBytes));
                for (int u = 0; u < ng; ++u) {
                    const uint32_t d_tmem = tmem + b * C::kBufCols + u * C::kAccCols + (side_b ? K : 0);
                    const uint64_t ad = sw128_desc(smem_u32(stage + (size_t)u * kTileBytes));
#pragma unroll
                    for (int k = 0; k < kChunkK / 16; ++k)
                        mma_bf16(d_tmem, ad + 2 * k, bd + 2 * k, idesc, (kk > 0 || k > 0) ? 1u : 0u);
                }
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
    } else if (!SL && (warp == 2 || warp == 3)) {
        // ---------------- sign generators (two warps, one half-row each)
        uint32_t ring = 0;
        bool ok = true;
        for (int ng; ok && (ng = it.take<G>(p, ncl, crank, gx, gt)) > 0;)
            for (int kc = 0; kc < nk_tot; ++kc, ++ring) {
                const int s = ring % C::kStages;
                const uint32_t ph = (ring / C::kStages) & 1u;
                const bool side_b = kc >= p.nk_in;
                const uint64_t key = side_b ? p.key_out : p.key_in;
                const uint64_t rb = (uint64_t)(side_b ? kc - p.nk_in : kc);
                // K = 128: each warp writes whole rows of one half of the K columns (columns
                // col0 and col0 + 32 per lane); their sign words and table expansion do not
                // depend on the stage's memory, so they are formed before the wait below
                const int col0 = (warp - 2) * (K / 2) + lane;
                uint4 q[C::kLut ? 2 : 1][8];
                if constexpr (C::kLut) {
                    const uint32_t lut = smem_u32(smem + C::kLutOff);
#pragma unroll
                    for (int j = 0; j < 2; ++j) expand_signs(q[j], sign_word(key, (uint32_t)(col0 + 32 * j), rb), lut);
                }
                bool got = true;
                if (lane == 0) got = wait_bounded(smem_u32(&empty[s]), ph ^ 1u, abort, p.err);
                got = __shfl_sync(0xffffffffu, got, 0);
                __syncwarp();
                if (!got) {
                    ok = false;
                    break;
                }
                uint8_t* tile = sA + (size_t)s * C::kStageBytes + (size_t)G * kTileBytes;
                if constexpr (C::kLut) {
#pragma unroll
                    for (int j = 0; j < 2; ++j) store_sign_row(tile, col0 + 32 * j, q[j]);
                } else {
                    for (int col = lane; col < K; col += 32)
                        write_sign_half(tile, col, sign_word(key, (uint32_t)col, rb), warp - 2);
                }
                fence_proxy_async();
                __syncwarp();
                if (lane == 0) mbar_arrive(smem_u32(&sready[s]));
            }
    } else if (C::kParted && warp >= 4) {
        // ---------------- epilogue, one example per tile (no packing): each tile's token
        // rows in parts of kStageRows (part h holds the TMEM lane quadrants of warps
        // h * kWarpsPer ..), each part staged in shared memory and contracted,
        // Phi += Bt^T At, in fp32. A warp releases the accumulator buffer once it has
        // read its quadrant of the group's last tile. The accumulators live for one
        // example (K = 128: the loop nest keeps them within 255 registers a thread).
        const int q = warp & 3;
        const int et = threadIdx.x - 128;
        const int rg = et >> 3, cg = et & 7;
        constexpr int kParts = kTileM / C::kStageRows, kWarpsPer = 4 / kParts;
        uint32_t grp = 0, red_use = 0;
        bool ok = true;
        int ng = it.take<G>(p, ncl, crank, gx, gt), u = 0;  // u: next tile of the current group
        while (ok && ng > 0) {
            const int64_t cur = gx[u];
            float acc[C::RB][C::CB];
#pragma unroll
            for (int a = 0; a < C::RB; ++a)
#pragma unroll
                for (int c = 0; c < C::CB; ++c) acc[a][c] = 0.f;
            do {
                const uint32_t b = grp & 1u, use = grp >> 1;
                if (u == 0) {
                    bool got = true;
                    if (lane == 0) got = wait_bounded(smem_u32(&tfull[b]), use & 1u, abort, p.err);
                    got = __shfl_sync(0xffffffffu, got, 0);
                    if (epi_any(!got)) {
                        ok = false;
                        break;
                    }
                    tc_fence_after();
                }
                const uint32_t tbase =
                    tmem + ((uint32_t)(q * 32) << 16) + b * C::kBufCols + (uint32_t)u * C::kAccCols;
                for (int h = 0; h < kParts; ++h) {
                    if (q / kWarpsPer == h) {
                        const int srow = (q % kWarpsPer) * 32 + lane;
#pragma unroll 4
                        for (int c0 = 0; c0 < 2 * K; c0 += 16) {
                            float v[16];
                            tmem_ld16(tbase + c0, v);
                            float* dst = c0 < K ? stX + srow * C::kStageLd + c0 : stY + srow * C::kStageLd + (c0 - K);
#pragma unroll
                            for (int i = 0; i < 16; i += 4)
                                *reinterpret_cast<float4*>(dst + i) = make_float4(v[i], v[i + 1], v[i + 2], v[i + 3]);
                        }
                        if (u == ng - 1) {
                            tc_fence_before();
                            __syncwarp();
                            if (lane == 0) mbar_arrive(smem_u32(&tempty[b]));
                        }
                    }
                    epi_sync();
#pragma unroll(K > 64 ? 1 : 4)
                    for (int t = 0; t < C::kStageRows; ++t) {
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
                if (++u == ng) {
                    ++grp;
                    ng = it.take<G>(p, ncl, crank, gx, gt);
                    u = 0;
                }
            } while (ng > 0 && gx[u] == cur);
            if constexpr (BAL) {
                if (ok) store_phi_bal<C>(acc, cur, p, et, abort + 1);
            } else if (ok && !store_phi<C>(acc, cur, p, crank, stX, red_go, red_full, red_use, abort, et, lane)) {
                ok = false;
            }
        }
    } else if (warp >= 4) {
        // ---------------- epilogue: TMEM -> shared -> Phi += Bt^T At
        const int q = warp & 3;          // TMEM lane quadrant of this warp
        const int et = threadIdx.x - 128;
        const int row = q * 32 + lane;   // token row within the tile
        const int rg = et >> 3, cg = et & 7;
        uint32_t grp = 0, red_use = 0;
        bool stop = false;
        int64_t cur = -1;                // example whose Phi is accumulating (pack == 1)
        float acc[C::RB][C::CB];
        // K-FAC factor covariances (unscaled signs): ca += At^T At, cgm += Bt^T Bt over valid rows
        float ca[KF ? C::RB : 1][KF ? C::CB : 1], cgm[KF ? C::RB : 1][KF ? C::CB : 1];
#pragma unroll
        for (int a = 0; a < C::RB; ++a)
#pragma unroll
            for (int c = 0; c < C::CB; ++c) acc[a][c] = 0.f;
        if constexpr (KF) {
#pragma unroll
            for (int a = 0; a < C::RB; ++a)
#pragma unroll
                for (int c = 0; c < C::CB; ++c) ca[a][c] = cgm[a][c] = 0.f;
        }

        // Phi of example `n` is complete in every cluster CTA: reduce the partial
        // blocks into the leader (rank 0) over distributed shared memory and
        // write it. The leader's staging buffer (free between tiles) receives
        // member r's partial at offset (r-1)*K*K, thread-major.
        auto flush = [&](int64_t n) -> bool {
            if (p.cs > 1) {
                constexpr int kPer = C::RB * C::CB;
                const uint32_t slot = smem_u32(stX) + (uint32_t)(et * kPer) * 4u;
                bool got = true;
                if (crank == 0) {
                    if (et == 0)
                        for (int r = 1; r < p.cs; ++r) mbar_arrive_remote(smem_u32(red_go), (uint32_t)r);
                    if (lane == 0) got = wait_bounded_cluster(smem_u32(red_full), red_use & 1u, abort, p.err);
                    got = __shfl_sync(0xffffffffu, got, 0);
                    if (epi_any(!got)) return false;
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
                    if (epi_any(!got)) return false;
                    const uint32_t dst = map_rank(slot, 0) + (crank - 1) * (uint32_t)(K * K) * 4u;
#pragma unroll
                    for (int a = 0; a < C::RB; ++a)
#pragma unroll
                        for (int c = 0; c < C::CB; ++c)
                            st_cluster_f32(dst + (uint32_t)(a * C::CB + c) * 4u, acc[a][c]);
                    fence_acq_rel_cluster();
                    epi_sync();
                    if (et == 0) mbar_arrive_remote(smem_u32(red_full), 0u);
                }
                ++red_use;
                if (crank != 0) return true;
            }
            float* out = p.phi + n * p.ld_phi;
#pragma unroll
            for (int a = 0; a < C::RB; ++a)
#pragma unroll
                for (int c = 0; c < C::CB; ++c) out[(rg * C::RB + a) * K + cg * C::CB + c] = acc[a][c] * p.scale;
            return true;
        };

        for (int ng; !stop && (ng = it.take<G>(p, ncl, crank, gx, gt)) > 0; ++grp) {
            const uint32_t b = grp & 1u, use = grp >> 1;
            bool got = true;
            if (lane == 0) got = wait_bounded(smem_u32(&tfull[b]), use & 1u, abort, p.err);
            got = __shfl_sync(0xffffffffu, got, 0);
            if (epi_any(!got)) {
                stop = true;
                break;
            }
            tc_fence_after();
            for (int u = 0; u < ng; ++u) {
                if (!FO && p.pack == 1 && gx[u] != cur) {
                    if (cur >= 0 && !flush(cur)) {
                        stop = true;
                        break;
                    }
                    cur = gx[u];
#pragma unroll
                    for (int a = 0; a < C::RB; ++a)
#pragma unroll
                        for (int c = 0; c < C::CB; ++c) acc[a][c] = 0.f;
                }
                const uint32_t tbase =
                    tmem + ((uint32_t)(q * 32) << 16) + b * C::kBufCols + (uint32_t)u * C::kAccCols;
#pragma unroll
                for (int c0 = 0; c0 < 2 * K; c0 += 16) {
                    float v[16];
                    tmem_ld16(tbase + c0, v);
                    float* dst = c0 < K ? stX + row * C::kStageLd + c0 : stY + row * C::kStageLd + (c0 - K);
#pragma unroll
                    for (int i = 0; i < 16; i += 4)
                        *reinterpret_cast<float4*>(dst + i) = make_float4(v[i], v[i + 1], v[i + 2], v[i + 3]);
                }
                if (u == ng - 1) {
                    tc_fence_before();
                    __syncwarp();
                    if (lane == 0) mbar_arrive(smem_u32(&tempty[b]));
                }
                epi_sync();
                if constexpr (FO) {
                    // token rows of this tile in the [N*T] row space: packed tiles hold pack*T
                    // consecutive rows, a long tile rows tt*128 .. of example x
                    int64_t g0;
                    int nrows;
                    if (p.pack > 1) {
                        g0 = gx[u] * p.pack * p.T;
                        nrows = p.pack * (int)p.T;
                    } else {
                        g0 = gx[u] * p.T + (int64_t)gt[u] * kTileM;
                        nrows = (int)(p.T - (int64_t)gt[u] * kTileM < kTileM ? p.T - (int64_t)gt[u] * kTileM : kTileM);
                    }
                    const int64_t lim = p.N * p.T - g0;
                    if (lim < nrows) nrows = (int)lim;
                    float* oa = p.fout + g0 * K;
                    float* ob = p.fout + p.N * p.T * K + g0 * K;
                    for (int idx = et; idx < nrows * (K / 4); idx += 128) {
                        const int r = idx / (K / 4), c4 = (idx - r * (K / 4)) * 4;
                        *reinterpret_cast<float4*>(oa + (int64_t)r * K + c4) =
                            *reinterpret_cast<const float4*>(stX + r * C::kStageLd + c4);
                        *reinterpret_cast<float4*>(ob + (int64_t)r * K + c4) =
                            *reinterpret_cast<const float4*>(stY + r * C::kStageLd + c4);
                    }
                    epi_sync();
                    continue;
                }
                if constexpr (KF) {
                    // rows of packed tiles past pack * T belong to the next tile's examples
                    const int rows = p.pack == 1 ? kTileM : p.pack * (int)p.T;
#pragma unroll 2
                    for (int t = 0; t < rows; ++t) {
                        float xa[C::RB], xc[C::CB], ya[C::RB], yc[C::CB];
#pragma unroll
                        for (int a = 0; a < C::RB; ++a) {
                            xa[a] = stX[t * C::kStageLd + rg * C::RB + a];
                            ya[a] = stY[t * C::kStageLd + rg * C::RB + a];
                        }
#pragma unroll
                        for (int c = 0; c < C::CB; ++c) {
                            xc[c] = stX[t * C::kStageLd + cg * C::CB + c];
                            yc[c] = stY[t * C::kStageLd + cg * C::CB + c];
                        }
#pragma unroll
                        for (int a = 0; a < C::RB; ++a)
#pragma unroll
                            for (int c = 0; c < C::CB; ++c) {
                                ca[a][c] = fmaf(xa[a], xc[c], ca[a][c]);
                                cgm[a][c] = fmaf(ya[a], yc[c], cgm[a][c]);
                            }
                    }
                }
                if (p.pack == 1) {
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
                } else {
                    // packed tile: example x * pack + j owns rows j*T .. j*T + T - 1
                    for (int j = 0; j < p.pack; ++j) {
                        const int64_t e = gx[u] * p.pack + j;
                        if (e >= p.N) break;
                        float a2[C::RB][C::CB];
#pragma unroll
                        for (int a = 0; a < C::RB; ++a)
#pragma unroll
                            for (int c = 0; c < C::CB; ++c) a2[a][c] = 0.f;
                        const int t1 = (j + 1) * (int)p.T;
#pragma unroll 4
                        for (int t = j * (int)p.T; t < t1; ++t) {
                            float y[C::RB], x[C::CB];
#pragma unroll
                            for (int a = 0; a < C::RB; ++a) y[a] = stY[t * C::kStageLd + rg * C::RB + a];
#pragma unroll
                            for (int c = 0; c < C::CB; ++c) x[c] = stX[t * C::kStageLd + cg * C::CB + c];
#pragma unroll
                            for (int a = 0; a < C::RB; ++a)
#pragma unroll
                                for (int c = 0; c < C::CB; ++c) a2[a][c] = fmaf(y[a], x[c], a2[a][c]);
                        }
                        float* out = p.phi + e * p.ld_phi;
#pragma unroll
                        for (int a = 0; a < C::RB; ++a)
#pragma unroll
                            for (int c = 0; c < C::CB; ++c)
                                out[(rg * C::RB + a) * K + cg * C::CB + c] = a2[a][c] * p.scale;
                    }
                }
                epi_sync();
            }
        }
        if (!FO && !stop && p.pack == 1 && cur >= 0) flush(cur);
        if constexpr (KF) {
            float* out = p.cov + (size_t)blockIdx.x * 2 * K * K;
#pragma unroll
            for (int a = 0; a < C::RB; ++a)
#pragma unroll
                for (int c = 0; c < C::CB; ++c) {
                    const int e = (rg * C::RB + a) * K + cg * C::CB + c;
                    out[e] = ca[a][c];
                    out[K * K + e] = cgm[a][c];
                }
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
// out-of-range elements read as zero. For packed tiles the same memory is viewed
// as [1][N*T][d], so one box spans several consecutive examples.
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

// A side's sign table for the SL kernel: tab[j][r] = S[r][j] as bf16 +-1 for
// r < d, j < K (bit r mod 64 of sign word (j, r / 64); a set bit is -1), the
// same signs the generator warps write. One thread per (column, 64-row group).
__global__ void sign_table_kernel(uint16_t* __restrict__ tab, int64_t d, int K, uint64_t key) {
    const int64_t groups = (d + 63) / 64;
    for (int64_t e = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; e < groups * K;
         e += (int64_t)gridDim.x * blockDim.x) {
        const int j = (int)(e / groups);
        const int64_t rb = e - (int64_t)j * groups;
        const uint64_t w = sign_word(key, (uint32_t)j, (uint64_t)rb);
        uint16_t* row = tab + (int64_t)j * d + rb * 64;
        const int64_t n = (d - rb * 64) < 64 ? (d - rb * 64) : 64;
        if (n == 64) {
#pragma unroll
            for (int c = 0; c < 8; ++c) {
                uint32_t q[4];
#pragma unroll
                for (int t = 0; t < 4; ++t) {
                    const uint32_t lo = 0x3F80u | ((uint32_t)((w >> (8 * c + 2 * t)) & 1u) << 15);
                    const uint32_t hi = 0x3F80u | ((uint32_t)((w >> (8 * c + 2 * t + 1)) & 1u) << 15);
                    q[t] = lo | (hi << 16);
                }
                *reinterpret_cast<uint4*>(row + 8 * c) = make_uint4(q[0], q[1], q[2], q[3]);
            }
        } else {
            for (int64_t r = 0; r < n; ++r) row[r] = (uint16_t)(0x3F80u | ((uint32_t)((w >> r) & 1u) << 15));
        }
    }
}

// 3-D map over a sign table [1][K][d] (bf16): box 64 (d) x K x 1, 128B swizzle, zero fill past d.
bool make_sign_map(CUtensorMap* tm, const void* tab, int64_t d, int K) {
    EncodeTiledFn enc = encode_fn();
    if (!enc) return false;
    cuuint64_t dims[3] = {(cuuint64_t)d, (cuuint64_t)K, 1};
    cuuint64_t strides[2] = {(cuuint64_t)(d * 2), (cuuint64_t)(K * d * 2)};
    cuuint32_t box[3] = {kChunkK, (cuuint32_t)K, 1};
    cuuint32_t estr[3] = {1, 1, 1};
    return enc(tm, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(tab), dims, strides, box, estr,
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

int device_sms() {
    static int sms = 0;
    if (!sms) {
        int dev = 0, n = 0;
        cudaGetDevice(&dev);
        cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev);
        sms = n > 0 ? n : 1;
    }
    return sms;
}

// SMs this launch may fill: all of them, or the tda_set_sm_budget cap
int sm_count() {
    const int sms = device_sms(), b = sm_budget();
    return (b > 0 && b < sms) ? b : sms;
}

template <int K, int G, bool KF, bool FO, bool SL = false, int SR = Cfg<K, G>::kStageRows, bool BAL = false>
cudaError_t launch_kg(const tda_layer_desc& L, const void* A, const void* B, int64_t N, float* phi,
                      int64_t ld_phi, unsigned int* err, cudaStream_t s, int pack, float* cov, int* grid_out,
                      float* fout, const void* signs = nullptr, void* bal_ws = nullptr) {
    using C = Cfg<K, G, SR, (K > 64) && !SL>;
    if (C::kParted && pack > 1) return cudaErrorInvalidValue;  // packed tiles are staged whole
    if (BAL && !bal_ws) return cudaErrorInvalidValue;
    CUtensorMap tmA, tmB, tmSA, tmSB;
    if constexpr (SL) {
        const uint16_t* tab = (const uint16_t*)signs;
        if (!make_sign_map(&tmSA, tab, L.d_in, K) || !make_sign_map(&tmSB, tab + (int64_t)K * L.d_in, L.d_out, K))
            return cudaErrorInvalidValue;
    } else {
        memset(&tmSA, 0, sizeof(tmSA));
        memset(&tmSB, 0, sizeof(tmSB));
    }
    if (pack > 1) {
        if (!make_map(&tmA, A, 1, N * L.T, L.d_in) || !make_map(&tmB, B, 1, N * L.T, L.d_out))
            return cudaErrorInvalidValue;
    } else if (!make_map(&tmA, A, N, L.T, L.d_in) || !make_map(&tmB, B, N, L.T, L.d_out)) {
        return cudaErrorInvalidValue;
    }
    Params p;
    p.N = N;
    p.T = L.T;
    p.d_in = L.d_in;
    p.d_out = L.d_out;
    p.ld_phi = ld_phi;
    p.pack = pack;
    p.n_slots = pack > 1 ? (N + pack - 1) / pack : N;
    p.key_in = side_key(L.seed, L.layer, 0);
    p.key_out = side_key(L.seed, L.layer, 1);
    p.scale = projection_scale(L);
    p.phi = phi;
    p.err = err;
    p.n_ttiles = pack > 1 ? 1 : (int)((L.T + kTileM - 1) / kTileM);
    p.nk_in = (int)((L.d_in + kChunkK - 1) / kChunkK);
    p.nk_out = (int)((L.d_out + kChunkK - 1) / kChunkK);
    p.cov = cov;
    p.fout = fout;
    p.n_units = p.n_slots * p.n_ttiles;
    p.part = nullptr;
    p.cnt = nullptr;
    const int sms = sm_count();
    cudaError_t e = smem_attr_once<project_tc_kernel<K, G, KF, FO, SL, SR, BAL>>((int)C::kSmem);
    if (e != cudaSuccess) return e;
    // Fewer examples than SMs: a cluster of cs CTAs shares each example's token
    // tiles and reduces the partial features through distributed shared memory.
    int cs = 1;
    if (!BAL && pack == 1 && N < sms && !FO) cs = (2 * N >= sms) ? 2 : 4;
    while (cs > 1 && (cs > p.n_ttiles || cs > C::kMaxCs)) cs >>= 1;
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
    cfg.gridDim = dim3((unsigned)(cs * (device_sms() / cs)));
    int max_clusters = max_clusters_once<project_tc_kernel<K, G, KF, FO, SL, SR, BAL>>(cfg, cs, sms / cs);
    if (max_clusters > sms / cs) max_clusters = sms / cs;  // the SM budget (the occupancy query sees every SM)
    int64_t clusters = (FO || BAL) ? p.n_units : p.n_slots;
    if (clusters > max_clusters) clusters = max_clusters;
    cfg.gridDim = dim3((unsigned)(clusters * cs));
    if (grid_out) *grid_out = (int)(clusters * cs);
    if constexpr (BAL) {
        // partial slots, then one counter per CTA (cleared here; each call leaves them clear)
        p.part = (float*)bal_ws;
        p.cnt = (unsigned int*)((char*)bal_ws + (size_t)2 * device_sms() * K * K * sizeof(float));
        e = cudaMemsetAsync(p.cnt, 0, (size_t)clusters * sizeof(unsigned int), s);
        if (e != cudaSuccess) return e;
    }
    note_launches(1);
    e = cudaLaunchKernelEx(&cfg, project_tc_kernel<K, G, KF, FO, SL, SR, BAL>, tmA, tmB, tmSA, tmSB, p);
    if (e != cudaSuccess) return e;
    return cudaGetLastError();
}

// Two tiles per stage once every CTA has at least two groups of work; fewer
// units run one tile per stage so that they spread over all SMs.
template <int K, bool KF, bool FO>
cudaError_t launch_k(const tda_layer_desc& L, const void* A, const void* B, int64_t N, float* phi,
                     int64_t ld_phi, unsigned int* err, cudaStream_t s, float* cov, int* grid_out, float* fout,
                     const void* signs = nullptr, void* bal_ws = nullptr) {
    // K = 128 keeps one example per tile (its epilogue contracts 64-row halves)
    int pack = (K <= 64 && L.T <= 64) ? (int)(kTileM / L.T) : 1;
    if (pack > 1) {
        // packed rows are addressed with 32-bit TMA coordinates and the [1][N*T][d]
        // view's outer stride must stay below 2^40 bytes: split larger batches
        const int64_t d_max = L.d_in > L.d_out ? L.d_in : L.d_out;
        int64_t max_n = ((int64_t)1 << 30) / L.T;
        const int64_t by_stride = (((int64_t)1 << 40) - 1) / (L.T * d_max * 2);
        if (by_stride < max_n) max_n = by_stride;
        max_n = max_n / pack * pack;
        if (max_n < pack) pack = 1;  // one example per tile instead
        else if (N > max_n) {
            if (KF || FO) return cudaErrorInvalidValue;  // one partial slab / one factor block per launch
            const size_t a_ex = (size_t)L.T * L.d_in * 2, b_ex = (size_t)L.T * L.d_out * 2;
            for (int64_t e0 = 0; e0 < N; e0 += max_n) {
                const int64_t n = N - e0 < max_n ? N - e0 : max_n;
                cudaError_t e = launch_k<K, KF, FO>(L, (const char*)A + e0 * a_ex, (const char*)B + e0 * b_ex, n,
                                                    phi + e0 * ld_phi, ld_phi, err, s, nullptr, nullptr, nullptr,
                                                    signs, bal_ws);
                if (e != cudaSuccess) return e;
            }
            return cudaSuccess;
        }
    }
    // With the balanced-range workspace (one example per tile): contiguous runs of token tiles
    // per CTA, 32 token rows staged at a time (room for one or two more stages in the ring).
    // Without it, at least one example per SM (no cluster shares an example) stages 32 rows as
    // well for k >= 64 (k <= 32 measured faster with whole tiles: 7.1-7.3 against 6.9 TB/s on
    // the Llama-1B block); fewer examples keep the larger staging rows, which hold the cluster's
    // partial blocks.
    const bool bal = bal_ws && pack == 1;
    const bool narrow = K >= 64 && pack == 1 && N >= (int64_t)sm_count();
    if constexpr (K > 64) {
        if constexpr (!KF && !FO) {
            if (signs) {
                if (bal)
                    return launch_kg<K, 1, false, false, true, 32, true>(L, A, B, N, phi, ld_phi, err, s, pack, cov,
                                                                         grid_out, fout, signs, bal_ws);
                return narrow ? launch_kg<K, 1, false, false, true, 32>(L, A, B, N, phi, ld_phi, err, s, pack, cov,
                                                                         grid_out, fout, signs)
                              : launch_kg<K, 1, false, false, true>(L, A, B, N, phi, ld_phi, err, s, pack, cov,
                                                                    grid_out, fout, signs);
            }
            if (bal)
                return launch_kg<K, 1, false, false, false, 32, true>(L, A, B, N, phi, ld_phi, err, s, pack, cov,
                                                                      grid_out, fout, nullptr, bal_ws);
            if (narrow)
                return launch_kg<K, 1, false, false, false, 32>(L, A, B, N, phi, ld_phi, err, s, pack, cov, grid_out,
                                                                fout);
        }
        return launch_kg<K, 1, KF, FO>(L, A, B, N, phi, ld_phi, err, s, pack, cov, grid_out, fout);
    } else {
        const int64_t units = pack > 1 ? (N + pack - 1) / pack : N * ((L.T + kTileM - 1) / kTileM);
        if (units >= 4 * (int64_t)sm_count()) {
            if constexpr (!KF && !FO) {
                if (bal)
                    return launch_kg<K, 2, false, false, false, 32, true>(L, A, B, N, phi, ld_phi, err, s, pack, cov,
                                                                          grid_out, fout, nullptr, bal_ws);
                if (narrow)
                    return launch_kg<K, 2, false, false, false, 32>(L, A, B, N, phi, ld_phi, err, s, pack, cov,
                                                                    grid_out, fout);
            }
            return launch_kg<K, 2, KF, FO>(L, A, B, N, phi, ld_phi, err, s, pack, cov, grid_out, fout);
        }
        if constexpr (!KF && !FO)
            if (bal)
                return launch_kg<K, 1, false, false, false, 32, true>(L, A, B, N, phi, ld_phi, err, s, pack, cov,
                                                                      grid_out, fout, nullptr, bal_ws);
        return launch_kg<K, 1, KF, FO>(L, A, B, N, phi, ld_phi, err, s, pack, cov, grid_out, fout);
    }
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

// The plain projection also runs k = 128 on the tensor cores (the fused K-FAC
// covariances and the factor output stay at k <= 64).
bool project_tc_plain_supported(const tda_layer_desc& L, const void* A, const void* B) {
    if (L.k_in == 128 && L.k_out == 128) {
        tda_layer_desc L64 = L;
        L64.k_in = L64.k_out = 64;
        return project_tc_supported(L64, A, B);
    }
    return project_tc_supported(L, A, B);
}

size_t project_tc_sign_table_bytes(const tda_layer_desc& L) {
    if (L.k_in != 128 || L.k_out != 128) return 0;
    return (size_t)L.k_in * (size_t)(L.d_in + L.d_out) * 2;
}

// Balanced token-tile ranges: two K x K partial blocks and one counter per SM.
size_t project_tc_balance_bytes(const tda_layer_desc& L) {
    const size_t sms = (size_t)device_sms();
    return sms * (2 * (size_t)L.k_in * L.k_out * sizeof(float) + sizeof(unsigned int));
}

size_t project_tc_ws_bytes(const tda_layer_desc& L) {
    return (project_tc_sign_table_bytes(L) + 255) / 256 * 256 + project_tc_balance_bytes(L);
}

cudaError_t launch_project_tc(const tda_layer_desc& L, const void* A, const void* B, int64_t N, float* phi,
                              int64_t ld_phi, unsigned int* err, cudaStream_t s, void* ws, size_t ws_bytes) {
    if (N == 0) return cudaSuccess;
    // ws (256-byte aligned): [k = 128: both sides' sign tables, rounded up to 256 bytes]
    // [balanced-range partials and counters]; either part is used when ws has room for it
    if (ws && ((uintptr_t)ws & 255)) ws = nullptr;
    const size_t sign_b = (project_tc_sign_table_bytes(L) + 255) / 256 * 256;
    void* bal_ws = (ws && ws_bytes >= project_tc_ws_bytes(L)) ? (char*)ws + sign_b : nullptr;
    switch (L.k_in) {
        case 16: return launch_k<16, false, false>(L, A, B, N, phi, ld_phi, err, s, nullptr, nullptr, nullptr, nullptr, bal_ws);
        case 32: return launch_k<32, false, false>(L, A, B, N, phi, ld_phi, err, s, nullptr, nullptr, nullptr, nullptr, bal_ws);
        case 64: return launch_k<64, false, false>(L, A, B, N, phi, ld_phi, err, s, nullptr, nullptr, nullptr, nullptr, bal_ws);
        case 128: {
            // with room in ws: both sides' sign tables once per call (L2-resident, read by TMA
            // beside the factor tiles) instead of sign tiles written by the generator warps
            const size_t need = project_tc_sign_table_bytes(L);
            const void* signs = nullptr;
            if (ws && ws_bytes >= need) {
                uint16_t* tab = (uint16_t*)ws;
                const int64_t items = 128 * ((L.d_in + 63) / 64 + (L.d_out + 63) / 64);
                const unsigned blocks = (unsigned)((items + 255) / 256 < 1216 ? (items + 255) / 256 : 1216);
                note_launches(2);
                sign_table_kernel<<<blocks, 256, 0, s>>>(tab, L.d_in, 128, side_key(L.seed, L.layer, 0));
                sign_table_kernel<<<blocks, 256, 0, s>>>(tab + 128 * L.d_in, L.d_out, 128,
                                                         side_key(L.seed, L.layer, 1));
                cudaError_t e = cudaGetLastError();
                if (e != cudaSuccess) return e;
                signs = tab;
            }
            return launch_k<128, false, false>(L, A, B, N, phi, ld_phi, err, s, nullptr, nullptr, nullptr, signs,
                                               bal_ws);
        }
        default: return cudaErrorNotSupported;
    }
}

// Projection plus K-FAC factor covariance partials: cov receives one slab of
// 2 * k * k floats per CTA (At^T At then Bt^T Bt, unscaled signs); *grid_out
// is the number of slabs written.
cudaError_t launch_project_tc_kfac(const tda_layer_desc& L, const void* A, const void* B, int64_t N, float* phi,
                                   int64_t ld_phi, float* cov, int* grid_out, unsigned int* err, cudaStream_t s) {
    *grid_out = 0;
    if (N == 0) return cudaSuccess;
    switch (L.k_in) {
        case 16: return launch_k<16, true, false>(L, A, B, N, phi, ld_phi, err, s, cov, grid_out, nullptr);
        case 32: return launch_k<32, true, false>(L, A, B, N, phi, ld_phi, err, s, cov, grid_out, nullptr);
        case 64: return launch_k<64, true, false>(L, A, B, N, phi, ld_phi, err, s, cov, grid_out, nullptr);
        default: return cudaErrorNotSupported;
    }
}

int project_tc_max_grid() { return device_sms(); }

// Projected factors of N examples (At rows then Bt rows, [N*T][k] each, fp32,
// unscaled signs) by the tensor-core kernel.
cudaError_t launch_project_factors_tc(const tda_layer_desc& L, const void* A, const void* B, int64_t N, float* Y,
                                      unsigned int* err, cudaStream_t s) {
    if (N == 0 || L.T == 0) return cudaSuccess;
    switch (L.k_in) {
        case 16: return launch_k<16, false, true>(L, A, B, N, nullptr, 0, err, s, nullptr, nullptr, Y);
        case 32: return launch_k<32, false, true>(L, A, B, N, nullptr, 0, err, s, nullptr, nullptr, Y);
        case 64: return launch_k<64, false, true>(L, A, B, N, nullptr, 0, err, s, nullptr, nullptr, Y);
        default: return cudaErrorNotSupported;
    }
}

}  // namespace tda
