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
#include <cuda_bf16.h>

#include "tda_internal.cuh"

namespace tda {
namespace {

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

constexpr int kMaskThreads = 512;
constexpr int kMaskPer = 32;  // coordinates per thread
constexpr int kMaskCoords = kMaskThreads * kMaskPer;

__device__ __forceinline__ float ldf(const float* p) { return *p; }
__device__ __forceinline__ float ldf(const __nv_bfloat16* p) { return __bfloat162float(*p); }

// out[n*ld_out + m] = sum_t B[n][t][rows[m]] * A[n][t][cols[m]] for the block's
// coordinates m; tokens staged tt at a time. Coordinates outside the layer give
// NaN. Needs d_in, d_out <= 65536 (a coordinate pair packs into 32 bits).
template <typename TF>
__global__ void __launch_bounds__(kMaskThreads)
mask_gather_kernel(const TF* __restrict__ A, const TF* __restrict__ B, int64_t T, int64_t d_in, int64_t d_out,
                   const int32_t* __restrict__ rows, const int32_t* __restrict__ cols, int64_t n_coords,
                   float* __restrict__ out, int64_t ld_out, int tt) {
    extern __shared__ unsigned char smraw[];
    TF* sa = (TF*)smraw;                    // [tt][d_in]
    TF* sb = sa + (int64_t)tt * d_in;       // [tt][d_out]
    const int64_t n = blockIdx.y;
    const int64_t m0 = (int64_t)blockIdx.x * kMaskCoords;
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
    for (int64_t t0 = 0; t0 < T; t0 += tt) {
        const int nt = (int)(T - t0 < tt ? T - t0 : tt);
        __syncthreads();
        for (int64_t x = threadIdx.x; x < (int64_t)nt * d_in; x += blockDim.x) sa[x] = An[t0 * d_in + x];
        for (int64_t x = threadIdx.x; x < (int64_t)nt * d_out; x += blockDim.x) sb[x] = Bn[t0 * d_out + x];
        __syncthreads();
        for (int t = 0; t < nt; ++t) {
            const TF* at = sa + (int64_t)t * d_in;
            const TF* bt = sb + (int64_t)t * d_out;
#pragma unroll
            for (int u = 0; u < kMaskPer; ++u) {
                const uint32_t v = rc[u] == 0xFFFFFFFFu ? 0u : rc[u];
                acc[u] = fmaf(ldf(bt + (v >> 16)), ldf(at + (v & 0xFFFFu)), acc[u]);
            }
        }
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
    const size_t smem = sizeof(float) * ((size_t)kTokTile * (ka + kg) + (size_t)ka * kg);
    cudaError_t e = cudaFuncSetAttribute(token_scores_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    note_launches(1);
    token_scores_kernel<<<dim3((unsigned)((T + kTokTile - 1) / kTokTile), (unsigned)n), 256, smem, s>>>(
        Ya, Yb, n, T, ka, kg, R, n_q, ld_R, scale, out, ld_q, i0, beta);
    return cudaGetLastError();
}

// tokens staged per pass so that both factor rows fit in 96 KiB of shared memory
int mask_gather_tokens_per_pass(int64_t d_in, int64_t d_out, size_t el) {
    const int64_t per = (d_in + d_out) * (int64_t)el;
    int64_t tt = (96 * 1024) / per;
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
    const size_t smem = (size_t)tt * (size_t)(L.d_in + L.d_out) * el;
    const dim3 grid((unsigned)((n_coords + kMaskCoords - 1) / kMaskCoords), (unsigned)N);
    note_launches(1);
    cudaError_t e;
    if (dt == TDA_F32) {
        e = cudaFuncSetAttribute(mask_gather_kernel<float>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
        if (e != cudaSuccess) return e;
        mask_gather_kernel<float><<<grid, kMaskThreads, smem, s>>>((const float*)A, (const float*)B, L.T, L.d_in,
                                                                   L.d_out, rows, cols, n_coords, out, ld_out, tt);
    } else {
        e = cudaFuncSetAttribute(mask_gather_kernel<__nv_bfloat16>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 (int)smem);
        if (e != cudaSuccess) return e;
        mask_gather_kernel<__nv_bfloat16><<<grid, kMaskThreads, smem, s>>>(
            (const __nv_bfloat16*)A, (const __nv_bfloat16*)B, L.T, L.d_in, L.d_out, rows, cols, n_coords, out, ld_out,
            tt);
    }
    return cudaGetLastError();
}

}  // namespace tda
