// k_tokens.cu -- two reuses of the captured factors.
//
// Token-level scores (token-level attribution appendix): with the query-side
// matrix R_j (k_out x k_in; the projected, possibly preconditioned query
// feature) the score of train example i decomposes over its tokens,
//   s_t = g~_t^T R_j a~_t,   sum_t s_t = <Phi_i, R_j>.
// The projected factors a~_t, g~_t come from the factor projection kernel; one
// CTA handles 64 tokens of one example against every query.
//
// Random-mask reduction (App. B.4's reduced representation): the entries of
// DW = sum_t g_t a_t^T at a given list of coordinates, gathered from the
// factors without forming DW. One CTA per (example, block of coordinates)
// streams the example's tokens through shared memory.
#include <cuda.h>
#include <cuda_bf16.h>

#include <type_traits>

#include "tda_internal.cuh"

namespace tda {
namespace {

#include "tc_ptx.cuh"

constexpr int kTokTile = 64;

// out[j*ld_q + i*T + t] = beta*out + scale * g~_t^T R_j a~_t
__global__ void __launch_bounds__(256)
token_scores_kernel(const float* __restrict__ Ya, const float* __restrict__ Yb, int64_t n, int64_t T, int ka, int kg,
                    const float* __restrict__ R, int64_t n_q, int64_t ld_R, float scale, float* __restrict__ out,
                    int64_t ld_q, int64_t i0, float beta) {
    extern __shared__ float sm[];  // a~ [64][ka], g~ [64][kg], R_j [kg][ka]
    float* sa = sm;
    float* sg = sa + kTokTile * ka;
    float* sr = sg + kTokTile * kg;
    const int64_t i = blockIdx.y;  // example within the chunk
    const int64_t t0 = (int64_t)blockIdx.x * kTokTile;
    const int nt = (int)(T - t0 < kTokTile ? T - t0 : kTokTile);
    for (int x = threadIdx.x; x < nt * ka; x += blockDim.x) sa[x] = Ya[(i * T + t0) * ka + x];
    for (int x = threadIdx.x; x < nt * kg; x += blockDim.x) sg[x] = Yb[(i * T + t0) * kg + x];
    const int tl = threadIdx.x >> 2, q = threadIdx.x & 3;  // token, quarter of R's rows
    for (int64_t j = 0; j < n_q; ++j) {
        __syncthreads();
        for (int x = threadIdx.x; x < kg * ka; x += blockDim.x) sr[x] = R[j * ld_R + x];
        __syncthreads();
        float s = 0.f;
        if (tl < nt) {
            const float* a = sa + tl * ka;
            const float* g = sg + tl * kg;
            for (int r = q; r < kg; r += 4) {
                float u = 0.f;
                const float* rr = sr + r * ka;
                for (int c = 0; c < ka; ++c) u = fmaf(rr[c], a[c], u);
                s = fmaf(g[r], u, s);
            }
        }
        s += __shfl_xor_sync(0xffffffffu, s, 1);
        s += __shfl_xor_sync(0xffffffffu, s, 2);
        if (q == 0 && tl < nt) {
            float* dst = out + j * ld_q + (i0 + i) * T + t0 + tl;
            *dst = beta == 0.f ? scale * s : beta * (*dst) + scale * s;
        }
    }
}

// k <= 64: one thread per token holds a~_t and g~_t in registers; R_j is read
// from shared memory as broadcasts (every thread of a warp reads the same row).
template <int K>
__global__ void __launch_bounds__(256)
token_scores_reg_kernel(const float* __restrict__ Ya, const float* __restrict__ Yb, int64_t T,
                        const float* __restrict__ R, int64_t n_q, int64_t ld_R, float scale, float* __restrict__ out,
                        int64_t ld_q, int64_t i0, float beta) {
    __shared__ __align__(16) float sr[K * K];
    const int64_t i = blockIdx.y;
    const int64_t t = (int64_t)blockIdx.x * 256 + threadIdx.x;
    const bool valid = t < T;
    float a[K], g[K];
#pragma unroll
    for (int c = 0; c < K; c += 4) {
        float4 va = make_float4(0.f, 0.f, 0.f, 0.f), vg = va;
        if (valid) {
            va = *reinterpret_cast<const float4*>(Ya + (i * T + t) * K + c);
            vg = *reinterpret_cast<const float4*>(Yb + (i * T + t) * K + c);
        }
        a[c] = va.x, a[c + 1] = va.y, a[c + 2] = va.z, a[c + 3] = va.w;
        g[c] = vg.x, g[c + 1] = vg.y, g[c + 2] = vg.z, g[c + 3] = vg.w;
    }
    for (int64_t j = 0; j < n_q; ++j) {
        __syncthreads();
        for (int x = threadIdx.x; x < K * K; x += 256) sr[x] = R[j * ld_R + x];
        __syncthreads();
        float s = 0.f;
#pragma unroll
        for (int r = 0; r < K; ++r) {
            float u = 0.f;
#pragma unroll
            for (int c = 0; c < K; c += 4) {
                const float4 rv = *reinterpret_cast<const float4*>(sr + r * K + c);
                u = fmaf(rv.x, a[c], u);
                u = fmaf(rv.y, a[c + 1], u);
                u = fmaf(rv.z, a[c + 2], u);
                u = fmaf(rv.w, a[c + 3], u);
            }
            s = fmaf(g[r], u, s);
        }
        if (valid) {
            float* dst = out + j * ld_q + (i0 + i) * T + t;
            *dst = beta == 0.f ? scale * s : beta * (*dst) + scale * s;
        }
    }
}

constexpr int kMaskThreads = 512;

__device__ __forceinline__ float ldf(const float* p) { return *p; }
__device__ __forceinline__ float ldf(const __nv_bfloat16* p) { return __bfloat162float(*p); }

__device__ __forceinline__ void bulk_load(uint32_t dst, const void* src, uint32_t bytes, uint32_t bar) {
    asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(dst),
                 "l"((uint64_t)src), "r"(bytes), "r"(bar)
                 : "memory");
}

// out[n*ld_out + m] = sum_t B[n][t][rows[m]] * A[n][t][cols[m]] for the block's
// coordinates m. Tokens stream through two shared-memory buffers of tt tokens
// each, filled by bulk copies (one thread issues them, an mbarrier counts the
// bytes) while the other buffer is being read. Coordinates outside the layer
// give NaN. Needs d_in, d_out <= 65536 (a coordinate pair packs into 32 bits).
template <typename TF, int kMaskPer>
__global__ void __launch_bounds__(kMaskThreads)
mask_gather_kernel(const TF* __restrict__ A, const TF* __restrict__ B, int64_t T, int64_t d_in, int64_t d_out,
                   const int32_t* __restrict__ rows, const int32_t* __restrict__ cols, int64_t n_coords,
                   float* __restrict__ out, int64_t ld_out, int tt, unsigned int* err) {
    extern __shared__ __align__(16) unsigned char smraw[];
    const int64_t buf_elems = (int64_t)tt * (d_in + d_out);
    __shared__ __align__(8) uint64_t full[2];
    __shared__ int abort_flag;
    const int64_t n = blockIdx.y;
    const int64_t m0 = (int64_t)blockIdx.x * kMaskThreads * kMaskPer;
    uint32_t rc[kMaskPer];  // row << 16 | col; all ones = no valid coordinate
    float acc[kMaskPer];
#pragma unroll
    for (int u = 0; u < kMaskPer; ++u) {
        const int64_t m = m0 + threadIdx.x + (int64_t)u * kMaskThreads;
        rc[u] = 0xFFFFFFFFu;
        if (m < n_coords) {
            const int32_t r = rows[m], c = cols[m];
            if (r >= 0 && r < d_out && c >= 0 && c < d_in) rc[u] = ((uint32_t)r << 16) | (uint32_t)c;
        }
        acc[u] = 0.f;
    }
    const TF* An = A + n * T * d_in;
    const TF* Bn = B + n * T * d_out;
    const int passes = (int)((T + tt - 1) / tt);
    auto issue = [&](int p) {  // one thread: tokens of pass p into buffer p & 1
        const int64_t t0 = (int64_t)p * tt;
        const int nt = (int)(T - t0 < tt ? T - t0 : tt);
        TF* sa = (TF*)smraw + (p & 1) * buf_elems;
        TF* sb = sa + (int64_t)tt * d_in;
        const uint32_t ba = (uint32_t)(nt * d_in * (int64_t)sizeof(TF)), bb = (uint32_t)(nt * d_out * (int64_t)sizeof(TF));
        const uint32_t bar = smem_u32(&full[p & 1]);
        mbar_arrive_tx(bar, ba + bb);
        bulk_load(smem_u32(sa), An + t0 * d_in, ba, bar);
        bulk_load(smem_u32(sb), Bn + t0 * d_out, bb, bar);
    };
    if (threadIdx.x == 0) {
        mbar_init(smem_u32(&full[0]), 1);
        mbar_init(smem_u32(&full[1]), 1);
        abort_flag = 0;
        fence_mbar_init();
    }
    __syncthreads();
    if (threadIdx.x == 0) issue(0);
    bool ok = true;
    int p = 0;
    for (; p < passes; ++p) {
        if (threadIdx.x == 0 && p + 1 < passes) {  // the other buffer was released by the last sync
            fence_proxy_async();
            issue(p + 1);
        }
        ok = wait_bounded(smem_u32(&full[p & 1]), (uint32_t)(p >> 1) & 1u, &abort_flag, err);
        if (!ok) break;
        const int64_t t0 = (int64_t)p * tt;
        const int nt = (int)(T - t0 < tt ? T - t0 : tt);
        const TF* sa = (const TF*)smraw + (p & 1) * buf_elems;
        const TF* sb = sa + (int64_t)tt * d_in;
        for (int t = 0; t < nt; ++t) {
            const TF* at = sa + (int64_t)t * d_in;
            const TF* bt = sb + (int64_t)t * d_out;
#pragma unroll
            for (int u = 0; u < kMaskPer; ++u) {
                const uint32_t v = rc[u] == 0xFFFFFFFFu ? 0u : rc[u];
                acc[u] = fmaf(ldf(bt + (v >> 16)), ldf(at + (v & 0xFFFFu)), acc[u]);
            }
        }
        __syncthreads();  // buffer p & 1 is free for pass p + 2
    }
    if (!ok) {
        // drain the copies of passes p and p + 1 that may still be landing (bounded)
        if (threadIdx.x == 0)
            for (int q = p; q < p + 2 && q < passes; ++q) {
                const uint64_t t0 = global_ns();
                while (!mbar_try_wait(smem_u32(&full[q & 1]), (uint32_t)(q >> 1) & 1u))
                    if (global_ns() - t0 > kTimeoutNs) break;
            }
        return;
    }
#pragma unroll
    for (int u = 0; u < kMaskPer; ++u) {
        const int64_t m = m0 + threadIdx.x + (int64_t)u * kMaskThreads;
        if (m < n_coords) out[n * ld_out + m] = rc[u] != 0xFFFFFFFFu ? acc[u] : __int_as_float(0x7fc00000);
    }
}

}  // namespace

cudaError_t launch_token_scores(const float* Ya, const float* Yb, int64_t n, int64_t T, int ka, int kg,
                                const float* R, int64_t n_q, int64_t ld_R, float scale, float* out, int64_t ld_q,
                                int64_t i0, float beta, cudaStream_t s) {
    if (n == 0 || T == 0 || n_q == 0) return cudaSuccess;
    const bool aligned = ((uintptr_t)R & 15) == 0 && (ld_R & 3) == 0 && ((uintptr_t)Ya & 15) == 0 &&
                         ((uintptr_t)Yb & 15) == 0;
    if (ka == kg && aligned && (ka == 16 || ka == 32 || ka == 64)) {
        const dim3 grid((unsigned)((T + 255) / 256), (unsigned)n);
        note_launches(1);
        if (ka == 16)
            token_scores_reg_kernel<16><<<grid, 256, 0, s>>>(Ya, Yb, T, R, n_q, ld_R, scale, out, ld_q, i0, beta);
        else if (ka == 32)
            token_scores_reg_kernel<32><<<grid, 256, 0, s>>>(Ya, Yb, T, R, n_q, ld_R, scale, out, ld_q, i0, beta);
        else
            token_scores_reg_kernel<64><<<grid, 256, 0, s>>>(Ya, Yb, T, R, n_q, ld_R, scale, out, ld_q, i0, beta);
        return cudaGetLastError();
    }
    const size_t smem = sizeof(float) * ((size_t)kTokTile * (ka + kg) + (size_t)ka * kg);
    cudaError_t e = cudaFuncSetAttribute(token_scores_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    note_launches(1);
    token_scores_kernel<<<dim3((unsigned)((T + kTokTile - 1) / kTokTile), (unsigned)n), 256, smem, s>>>(
        Ya, Yb, n, T, ka, kg, R, n_q, ld_R, scale, out, ld_q, i0, beta);
    return cudaGetLastError();
}

// tokens per buffer so that two buffers of both factor rows fit in 96 KiB
int mask_gather_tokens_per_pass(int64_t d_in, int64_t d_out, size_t el) {
    const int64_t per = (d_in + d_out) * (int64_t)el;
    int64_t tt = (48 * 1024) / per;
    if (tt > 32) tt = 32;
    return (int)tt;
}

cudaError_t launch_mask_gather(const tda_layer_desc& L, tda_dtype dt, const void* A, const void* B, int64_t N,
                               const int32_t* rows, const int32_t* cols, int64_t n_coords, float* out, int64_t ld_out,
                               cudaStream_t s) {
    if (N == 0 || n_coords == 0) return cudaSuccess;
    const size_t el = dt == TDA_F32 ? 4 : 2;
    const int tt = mask_gather_tokens_per_pass(L.d_in, L.d_out, el);
    if (tt < 1) return cudaErrorInvalidValue;
    const size_t smem = 2 * (size_t)tt * (size_t)(L.d_in + L.d_out) * el;
    unsigned int* err = device_error_word();
    if (!err) return cudaErrorInvalidValue;
    int per = 32;  // coordinates per thread: the fewest that cover n_coords in one block, at most 32
    for (int c : {4, 8, 16})
        if (n_coords <= (int64_t)kMaskThreads * c) {
            per = c;
            break;
        }
    const dim3 grid((unsigned)((n_coords + (int64_t)kMaskThreads * per - 1) / ((int64_t)kMaskThreads * per)),
                    (unsigned)N);
    note_launches(1);
    cudaError_t e = cudaSuccess;
    auto go = [&](auto tf, auto pc) {
        using TF = decltype(tf);
        constexpr int P = decltype(pc)::value;
        e = cudaFuncSetAttribute(mask_gather_kernel<TF, P>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
        if (e != cudaSuccess) return;
        mask_gather_kernel<TF, P><<<grid, kMaskThreads, smem, s>>>((const TF*)A, (const TF*)B, L.T, L.d_in, L.d_out,
                                                                   rows, cols, n_coords, out, ld_out, tt, err);
    };
    using I4 = std::integral_constant<int, 4>;
    using I8 = std::integral_constant<int, 8>;
    using I16 = std::integral_constant<int, 16>;
    using I32 = std::integral_constant<int, 32>;
    if (dt == TDA_F32) {
        if (per == 4) go(0.f, I4{}); else if (per == 8) go(0.f, I8{}); else if (per == 16) go(0.f, I16{}); else go(0.f, I32{});
    } else {
        const __nv_bfloat16 z{};
        if (per == 4) go(z, I4{}); else if (per == 8) go(z, I8{}); else if (per == 16) go(z, I16{}); else go(z, I32{});
    }
    if (e != cudaSuccess) return e;
    return cudaGetLastError();
}

}  // namespace tda
