// k_routes.cu -- the materialised route (b) and the factorised Gram route (c)
// (Sec. 3.2 "FLOP-aware routing", App. A.4, Table 2), CUDA-core versions.
//
// Route (b): G = DW = g a^T, G[r][c] = sum_t B[t][r] A[t][c] (Eq. 1), then
//   projection: Phi = scale * S_out^T G S_in   (same result as Eq. 2), or
//   exact similarity: <G_q, G_i>_F.
// Route (c): <DW_q, DW_i>_F = sum_{t,s} <a_t^q, a_s^i> <g_t^q, g_s^i> (Eq. 4),
//   never forming DW.
#include <cuda_bf16.h>

#include <type_traits>

#include "tda_internal.cuh"

namespace tda {
namespace {

constexpr int kT = 64;   // tile edge
constexpr int kK = 32;   // contraction chunk
constexpr int kTh = 256;

__device__ __forceinline__ float ld1(const float* p) { return __ldg(p); }
__device__ __forceinline__ float ld1(const __nv_bfloat16* p) { return __bfloat162float(*p); }

// Batched G_e = B_e^T A_e for examples e in [e0, e0+nb); G row-major d_out x d_in.
template <typename T>
__global__ void __launch_bounds__(kTh)
materialize_kernel(const T* __restrict__ A, const T* __restrict__ B, int64_t e0, int64_t Tn,
                   int64_t d_in, int64_t d_out, float* __restrict__ G) {
    __shared__ float Bs[kK][kT + 1];
    __shared__ float As[kK][kT + 1];
    const int64_t e = e0 + blockIdx.z;
    const T* Ae = A + e * Tn * d_in;
    const T* Be = B + e * Tn * d_out;
    float* Ge = G + (int64_t)blockIdx.z * d_out * d_in;
    const int64_t r0 = (int64_t)blockIdx.y * kT, c0 = (int64_t)blockIdx.x * kT;
    const int tid = threadIdx.x, ty = tid / 16, tx = tid % 16;
    float acc[4][4] = {};
    for (int64_t t0 = 0; t0 < Tn; t0 += kK) {
        for (int x = tid; x < kK * kT; x += kTh) {
            const int tt = x / kT, cc = x % kT;
            const int64_t t = t0 + tt;
            Bs[tt][cc] = (t < Tn && r0 + cc < d_out) ? ld1(Be + t * d_out + r0 + cc) : 0.f;
            As[tt][cc] = (t < Tn && c0 + cc < d_in) ? ld1(Ae + t * d_in + c0 + cc) : 0.f;
        }
        __syncthreads();
#pragma unroll 8
        for (int tt = 0; tt < kK; ++tt)
#pragma unroll
            for (int u = 0; u < 4; ++u)
#pragma unroll
                for (int v = 0; v < 4; ++v)
                    acc[u][v] = fmaf(Bs[tt][ty * 4 + u], As[tt][tx * 4 + v], acc[u][v]);
        __syncthreads();
    }
#pragma unroll
    for (int u = 0; u < 4; ++u)
#pragma unroll
        for (int v = 0; v < 4; ++v) {
            const int64_t r = r0 + ty * 4 + u, c = c0 + tx * 4 + v;
            if (r < d_out && c < d_in) Ge[r * d_in + c] = acc[u][v];
        }
}

__device__ __forceinline__ float signed_term(uint64_t w, int bit, float v) {
    return ((w >> bit) & 1u) ? -v : v;
}

// X_e[r][j] = sum_c G_e[r][c] S_in[c][j]   (rows r of d_out, columns j of k_in)
__global__ void __launch_bounds__(kTh)
sign_right_kernel(const float* __restrict__ G, int64_t d_out, int64_t d_in, int k_in,
                  uint64_t key, int kind, float* __restrict__ X) {
    __shared__ float Gs[kT][kT + 1];  // [r][c]
    __shared__ uint64_t Ws[kT];
    const float* Ge = G + (int64_t)blockIdx.z * d_out * d_in;
    float* Xe = X + (int64_t)blockIdx.z * d_out * k_in;
    const int64_t r0 = (int64_t)blockIdx.y * kT;
    const int j0 = blockIdx.x * kT;
    const int tid = threadIdx.x, ty = tid / 16, tx = tid % 16;
    float acc[4][4] = {};
    for (int64_t c0 = 0; c0 < d_in; c0 += kT) {
        for (int x = tid; x < kT * kT; x += kTh) {
            const int rr = x / kT, cc = x % kT;
            Gs[rr][cc] = (r0 + rr < d_out && c0 + cc < d_in) ? Ge[(r0 + rr) * d_in + c0 + cc] : 0.f;
        }
        if (tid < kT) Ws[tid] = sign_word(key, (uint32_t)(j0 + tid), (uint64_t)(c0 >> 6));
        __syncthreads();
        if (kind == TDA_PROJ_RADEMACHER) {
            uint64_t w[4];
#pragma unroll
            for (int v = 0; v < 4; ++v) w[v] = Ws[tx * 4 + v];
            for (int cc = 0; cc < kT; ++cc)
#pragma unroll
                for (int u = 0; u < 4; ++u) {
                    const float g = Gs[ty * 4 + u][cc];
#pragma unroll
                    for (int v = 0; v < 4; ++v) acc[u][v] += signed_term(w[v], cc, g);
                }
        } else {
#pragma unroll
            for (int v = 0; v < 4; ++v) {
                const int64_t j = j0 + tx * 4 + v;
                if (j >= c0 && j < c0 + kT)
#pragma unroll
                    for (int u = 0; u < 4; ++u) acc[u][v] += Gs[ty * 4 + u][j - c0];
            }
        }
        __syncthreads();
    }
#pragma unroll
    for (int u = 0; u < 4; ++u)
#pragma unroll
        for (int v = 0; v < 4; ++v) {
            const int64_t r = r0 + ty * 4 + u;
            const int j = j0 + tx * 4 + v;
            if (r < d_out && j < k_in) Xe[r * k_in + j] = acc[u][v];
        }
}

// Phi_e[i][j] = scale * sum_r S_out[r][i] X_e[r][j]
__global__ void __launch_bounds__(kTh)
sign_left_kernel(const float* __restrict__ X, int64_t d_out, int k_in, int k_out, uint64_t key,
                 int kind, float scale, int64_t e0, float* __restrict__ phi, int64_t ld_phi) {
    __shared__ float Xs[kT][kT + 1];  // [r][j]
    __shared__ uint64_t Ws[kT];
    const float* Xe = X + (int64_t)blockIdx.z * d_out * k_in;
    const int i0 = blockIdx.y * kT, j0 = blockIdx.x * kT;
    const int tid = threadIdx.x, ty = tid / 16, tx = tid % 16;
    float acc[4][4] = {};
    for (int64_t rb = 0; rb < d_out; rb += kT) {
        for (int x = tid; x < kT * kT; x += kTh) {
            const int rr = x / kT, jj = x % kT;
            Xs[rr][jj] = (rb + rr < d_out && j0 + jj < k_in) ? Xe[(rb + rr) * k_in + j0 + jj] : 0.f;
        }
        if (tid < kT) Ws[tid] = sign_word(key, (uint32_t)(i0 + tid), (uint64_t)(rb >> 6));
        __syncthreads();
        if (kind == TDA_PROJ_RADEMACHER) {
            uint64_t w[4];
#pragma unroll
            for (int u = 0; u < 4; ++u) w[u] = Ws[ty * 4 + u];
            for (int rr = 0; rr < kT; ++rr)
#pragma unroll
                for (int v = 0; v < 4; ++v) {
                    const float x = Xs[rr][tx * 4 + v];
#pragma unroll
                    for (int u = 0; u < 4; ++u) acc[u][v] += signed_term(w[u], rr, x);
                }
        } else {
#pragma unroll
            for (int u = 0; u < 4; ++u) {
                const int64_t i = i0 + ty * 4 + u;
                if (i >= rb && i < rb + kT)
#pragma unroll
                    for (int v = 0; v < 4; ++v) acc[u][v] += Xs[i - rb][tx * 4 + v];
            }
        }
        __syncthreads();
    }
    const int64_t e = e0 + blockIdx.z;
#pragma unroll
    for (int u = 0; u < 4; ++u)
#pragma unroll
        for (int v = 0; v < 4; ++v) {
            const int i = i0 + ty * 4 + u, j = j0 + tx * 4 + v;
            if (i < k_out && j < k_in) phi[e * ld_phi + (int64_t)i * k_in + j] = acc[u][v] * scale;
        }
}

// Route (c): one CTA per (train i, query q) pair, 16x16 token tiles; each
// thread owns one (t, s) pair of the tile and forms <a_t,a_s> <g_t,g_s>.
template <typename T>
__global__ void __launch_bounds__(kTh)
gram_kernel(const T* __restrict__ Aq, const T* __restrict__ Bq, const T* __restrict__ At,
            const T* __restrict__ Bt, int64_t Tn, int64_t d_in, int64_t d_out,
            float* __restrict__ S, int64_t ld_S, float beta, float alpha, int self_pairs) {
    constexpr int TT = 16, KC = 64;
    __shared__ float Xq[TT][KC + 1];
    __shared__ float Xi[TT][KC + 1];
    __shared__ float red[kTh];
    const int64_t i = blockIdx.x, q = self_pairs ? blockIdx.x : blockIdx.y;  // self: <DW_i, DW_i>
    const int tid = threadIdx.x, tl = tid / TT, sl = tid % TT;
    float total = 0.f;
    for (int64_t t0 = 0; t0 < Tn; t0 += TT) {
        for (int64_t s0 = 0; s0 < Tn; s0 += TT) {
            float dots[2];
            for (int side = 0; side < 2; ++side) {
                const int64_t d = side == 0 ? d_in : d_out;
                const T* xq = (side == 0 ? Aq + q * Tn * d_in : Bq + q * Tn * d_out);
                const T* xi = (side == 0 ? At + i * Tn * d_in : Bt + i * Tn * d_out);
                float acc = 0.f;
                for (int64_t c0 = 0; c0 < d; c0 += KC) {
                    for (int x = tid; x < TT * KC; x += kTh) {
                        const int rr = x / KC, cc = x % KC;
                        const int64_t c = c0 + cc;
                        Xq[rr][cc] = (t0 + rr < Tn && c < d) ? ld1(xq + (t0 + rr) * d + c) : 0.f;
                        Xi[rr][cc] = (s0 + rr < Tn && c < d) ? ld1(xi + (s0 + rr) * d + c) : 0.f;
                    }
                    __syncthreads();
#pragma unroll 16
                    for (int cc = 0; cc < KC; ++cc) acc = fmaf(Xq[tl][cc], Xi[sl][cc], acc);
                    __syncthreads();
                }
                dots[side] = acc;
            }
            total = fmaf(dots[0], dots[1], total);
        }
    }
    red[tid] = total;
    __syncthreads();
    for (int w = kTh / 2; w > 0; w >>= 1) {
        if (tid < w) red[tid] += red[tid + w];
        __syncthreads();
    }
    if (tid == 0) {
        float* dst = S + q * ld_S + i;
        *dst = (beta == 0.f) ? alpha * red[0] : beta * (*dst) + alpha * red[0];
    }
}

// Projected factors of examples [e0, e0+n): At[e][t][j] = sum_c A[t][c] S_in[c][j],
// Bt[e][t][i] = sum_r B[t][r] S_out[r][i] (fp32, unscaled signs). One CTA per
// (example, 64-token chunk); thread (t = tid/4, 16 columns at (tid%4)*16).
template <typename T>
__global__ void __launch_bounds__(kTh)
project_factors_kernel(const T* __restrict__ X, int64_t e0, int64_t Tn, int64_t d, int k, uint64_t key,
                       int kind, float* __restrict__ Y) {
    __shared__ float Xs[64][kT + 1];  // 64 tokens x 64 features
    __shared__ uint64_t Ws[256];
    const int64_t e = e0 + blockIdx.y;
    const int64_t t0 = (int64_t)blockIdx.x * 64;
    const T* Xe = X + e * Tn * d;
    float* Ye = Y + (int64_t)blockIdx.y * Tn * k;
    const int tid = threadIdx.x, tl = tid >> 2, cq = (tid & 3) * 16;
    for (int j0 = 0; j0 < k; j0 += 64) {
        float acc[16];
#pragma unroll
        for (int q = 0; q < 16; ++q) acc[q] = 0.f;
        for (int64_t c0 = 0; c0 < d; c0 += kT) {
            __syncthreads();
            for (int x = tid; x < 64 * kT; x += kTh) {
                const int tt = x / kT, cc = x % kT;
                Xs[tt][cc] = (t0 + tt < Tn && c0 + cc < d) ? ld1(Xe + (t0 + tt) * d + c0 + cc) : 0.f;
            }
            if (tid < 64) Ws[tid] = sign_word(key, (uint32_t)(j0 + tid), (uint64_t)(c0 >> 6));
            __syncthreads();
            if (kind == TDA_PROJ_RADEMACHER) {
                for (int cc = 0; cc < kT; ++cc) {
                    const float v = Xs[tl][cc];
#pragma unroll
                    for (int q = 0; q < 16; ++q) acc[q] += signed_term(Ws[cq + q], cc, v);
                }
            } else {
#pragma unroll
                for (int q = 0; q < 16; ++q) {
                    const int64_t j = j0 + cq + q;
                    if (j >= c0 && j < c0 + kT) acc[q] += Xs[tl][j - c0];
                }
            }
        }
        if (t0 + tl < Tn)
#pragma unroll
            for (int q = 0; q < 16; ++q)
                if (j0 + cq + q < k) Ye[(t0 + tl) * k + j0 + cq + q] = acc[q];
    }
}

template <typename T>
void launch_materialize(const void* A, const void* B, int64_t e0, int64_t nb,
                        const tda_layer_desc& L, float* G, cudaStream_t s) {
    if constexpr (std::is_same<T, __nv_bfloat16>::value) {
        // bf16 factors: the tensor-core kernel (fp32 accumulation, same result up to summation order)
        unsigned int* err = device_error_word();
        if (err && materialize_tc_supported(L, TDA_BF16, A, B, G)) {
            launch_materialize_tc(L, A, B, e0, nb, G, err, s);
            return;
        }
    }
    dim3 grid((unsigned)((L.d_in + kT - 1) / kT), (unsigned)((L.d_out + kT - 1) / kT), (unsigned)nb);
    note_launches(1);
    materialize_kernel<T><<<grid, kTh, 0, s>>>((const T*)A, (const T*)B, e0, L.T, L.d_in, L.d_out, G);
}

}  // namespace

size_t materialize_ws_bytes_per_example(const tda_layer_desc& L) {
    return sizeof(float) * (size_t)(L.d_out * L.d_in + L.d_out * (int64_t)L.k_in);
}

cudaError_t launch_project_materialized(const tda_layer_desc& L, tda_dtype dt, const void* A,
                                        const void* B, int64_t N, float* phi, int64_t ld_phi,
                                        void* ws, size_t ws_bytes, cudaStream_t s) {
    const size_t per = materialize_ws_bytes_per_example(L);
    int64_t nb = (int64_t)(ws_bytes / per);
    if (nb < 1) return cudaErrorInvalidValue;
    if (nb > 65535) nb = 65535;
    const uint64_t key_in = side_key(L.seed, L.layer, 0);
    const uint64_t key_out = side_key(L.seed, L.layer, 1);
    const float scale = projection_scale(L);
    for (int64_t e0 = 0; e0 < N; e0 += nb) {
        const int64_t cnt = (N - e0) < nb ? (N - e0) : nb;
        float* G = (float*)ws;
        float* X = G + cnt * L.d_out * L.d_in;
        if (dt == TDA_BF16)
            launch_materialize<__nv_bfloat16>(A, B, e0, cnt, L, G, s);
        else
            launch_materialize<float>(A, B, e0, cnt, L, G, s);
        dim3 g2((unsigned)((L.k_in + kT - 1) / kT), (unsigned)((L.d_out + kT - 1) / kT), (unsigned)cnt);
        note_launches(2);
        sign_right_kernel<<<g2, kTh, 0, s>>>(G, L.d_out, L.d_in, L.k_in, key_in, L.kind, X);
        dim3 g3((unsigned)((L.k_in + kT - 1) / kT), (unsigned)((L.k_out + kT - 1) / kT), (unsigned)cnt);
        sign_left_kernel<<<g3, kTh, 0, s>>>(X, L.d_out, L.k_in, L.k_out, key_out, L.kind, scale, e0,
                                            phi, ld_phi);
        cudaError_t e = cudaGetLastError();
        if (e != cudaSuccess) return e;
    }
    return cudaSuccess;
}

// The Frobenius dots' split-K partial sums (at most 256 feature slices per query x train pair of a
// chunk) sit after the query and train gradients, so that even the smallest workspace (one train
// gradient at a time) keeps the feature axis split: one unsplit row of millions of features
// accumulated in the tensor pipe's truncating fp32 loses about 1e-2 of relative accuracy.
static size_t simexact_part_floats(int64_t n_q, int64_t chunk) { return (size_t)256 * (size_t)(n_q * chunk); }

size_t similarity_materialize_ws_bytes(const tda_layer_desc& L, int64_t n_q, int64_t chunk) {
    return sizeof(float) * ((size_t)((n_q + chunk) * L.d_out * L.d_in) + simexact_part_floats(n_q, chunk));
}

cudaError_t launch_similarity_materialized(const tda_layer_desc& L, tda_dtype dt, const void* Aq,
                                           const void* Bq, int64_t n_q, const void* At,
                                           const void* Bt, int64_t n_t, float* S, int64_t ld_S,
                                           float beta, void* ws, size_t ws_bytes, cudaStream_t s) {
    const int64_t gsz = L.d_out * L.d_in;
    const int64_t room = (int64_t)(ws_bytes / (sizeof(float) * (size_t)gsz)) - n_q;
    if (room < 1) return cudaErrorInvalidValue;
    int64_t chunk = room < 65535 ? room : 65535;
    float* Gq = (float*)ws;
    float* Gt = Gq + n_q * gsz;
    // The Frobenius dots have few rows and very long ones: split the feature
    // axis over many CTAs when the chunk leaves one train gradient's room for
    // the partial sums.
    // (3xTF32 tensor cores when the operands allow, decided once for every chunk:
    // Gq and Gt share base alignment and row length; fp32 factors keep fp32 CUDA-core
    // dots: the tensor pipe accumulates a slice of thousands of features in truncating
    // fp32, about 1e-5 of relative error, the size of the fp32 tolerance itself)
    const bool tc = dt == TDA_BF16 && score_dots_tc(Gq, n_q, gsz, Gt, chunk, gsz, gsz);
    int splits = score_splitk_splits(n_q, chunk, gsz, tc);
    float* part = nullptr;
    if (splits > 1) {
        const size_t need = (size_t)splits * (size_t)n_q * (size_t)chunk;
        const size_t grads = (size_t)(n_q + chunk) * (size_t)gsz;  // floats of the query and train DW
        if (ws_bytes / sizeof(float) >= grads + need) {
            part = Gq + grads;  // the partials' room after the train gradients
        } else if (chunk > 1 && need <= (size_t)gsz) {
            --chunk;
            part = Gt + chunk * gsz;
        } else {
            splits = 1;
        }
    }
    for (int64_t q0 = 0; q0 < n_q; q0 += 65535) {
        const int64_t cnt = (n_q - q0) < 65535 ? (n_q - q0) : 65535;
        if (dt == TDA_BF16)
            launch_materialize<__nv_bfloat16>(Aq, Bq, q0, cnt, L, Gq + q0 * gsz, s);
        else
            launch_materialize<float>(Aq, Bq, q0, cnt, L, Gq + q0 * gsz, s);
    }
    for (int64_t i0 = 0; i0 < n_t; i0 += chunk) {
        const int64_t cnt = (n_t - i0) < chunk ? (n_t - i0) : chunk;
        if (dt == TDA_BF16)
            launch_materialize<__nv_bfloat16>(At, Bt, i0, cnt, L, Gt, s);
        else
            launch_materialize<float>(At, Bt, i0, cnt, L, Gt, s);
        cudaError_t e = launch_score_splitk(Gq, n_q, gsz, Gt, cnt, gsz, gsz, S + i0, ld_S, beta, splits, part, tc, s);
        if (e != cudaSuccess) return e;
    }
    return cudaGetLastError();
}

cudaError_t launch_similarity_gram(const tda_layer_desc& L, tda_dtype dt, const void* Aq,
                                   const void* Bq, int64_t n_q, const void* At, const void* Bt,
                                   int64_t n_t, float* S, int64_t ld_S, float beta,
                                   cudaStream_t s) {
    if (n_q == 0 || n_t == 0) return cudaSuccess;
    dim3 grid((unsigned)n_t, (unsigned)n_q);
    note_launches(1);
    if (dt == TDA_BF16)
        gram_kernel<__nv_bfloat16><<<grid, kTh, 0, s>>>(
            (const __nv_bfloat16*)Aq, (const __nv_bfloat16*)Bq, (const __nv_bfloat16*)At,
            (const __nv_bfloat16*)Bt, L.T, L.d_in, L.d_out, S, ld_S, beta, 1.f, 0);
    else
        gram_kernel<float><<<grid, kTh, 0, s>>>((const float*)Aq, (const float*)Bq, (const float*)At,
                                                (const float*)Bt, L.T, L.d_in, L.d_out, S, ld_S, beta, 1.f, 0);
    return cudaGetLastError();
}

size_t project_factors_bytes_per_example(const tda_layer_desc& L) {
    return sizeof(float) * (size_t)(L.T * ((int64_t)L.k_in + L.k_out));
}

// Projected factors of n examples into Y: At block (n x T x k_in) then Bt block.
cudaError_t launch_project_factors(const tda_layer_desc& L, tda_dtype dt, const void* A, const void* B, int64_t e0,
                                   int64_t n, float* Y, cudaStream_t s) {
    if (n == 0 || L.T == 0) return cudaSuccess;
    if (dt == TDA_BF16) {
        // bf16 factors in the tensor-core kernel's shapes: the same projection, at HBM speed
        const void* Ae = (const char*)A + (size_t)e0 * L.T * L.d_in * 2;
        const void* Be = (const char*)B + (size_t)e0 * L.T * L.d_out * 2;
        unsigned int* err = device_error_word();
        if (err && project_tc_supported(L, Ae, Be) && ((uintptr_t)Y & 15) == 0 && n * L.T < (1LL << 30)) {
            cudaError_t e = launch_project_factors_tc(L, Ae, Be, n, Y, err, s);
            if (e != cudaErrorInvalidValue) return e;
        }
    }
    const uint64_t key_in = side_key(L.seed, L.layer, 0), key_out = side_key(L.seed, L.layer, 1);
    float* Ya = Y;
    float* Yb = Y + n * L.T * L.k_in;
    dim3 grid((unsigned)((L.T + 63) / 64), (unsigned)n);
    note_launches(2);
    if (dt == TDA_BF16) {
        project_factors_kernel<__nv_bfloat16><<<grid, kTh, 0, s>>>((const __nv_bfloat16*)A, e0, L.T, L.d_in, L.k_in,
                                                                   key_in, L.kind, Ya);
        project_factors_kernel<__nv_bfloat16><<<grid, kTh, 0, s>>>((const __nv_bfloat16*)B, e0, L.T, L.d_out,
                                                                   L.k_out, key_out, L.kind, Yb);
    } else {
        project_factors_kernel<float><<<grid, kTh, 0, s>>>((const float*)A, e0, L.T, L.d_in, L.k_in, key_in, L.kind, Ya);
        project_factors_kernel<float><<<grid, kTh, 0, s>>>((const float*)B, e0, L.T, L.d_out, L.k_out, key_out, L.kind,
                                                           Yb);
    }
    return cudaGetLastError();
}

// Eq. 4 on projected factors: S = beta*S + scale^2 * sum_{t,s} <a~,a~><g~,g~>.
cudaError_t launch_gram_projected(const tda_layer_desc& L, const float* Yq, int64_t n_q, const float* Yt,
                                  int64_t n_t, float* S, int64_t ld_S, float beta, cudaStream_t s) {
    if (n_q == 0 || n_t == 0) return cudaSuccess;
    const float sc = projection_scale(L);
    dim3 grid((unsigned)n_t, (unsigned)n_q);
    note_launches(1);
    gram_kernel<float><<<grid, kTh, 0, s>>>(Yq, Yq + n_q * L.T * L.k_in, Yt, Yt + n_t * L.T * L.k_in, L.T, L.k_in,
                                            L.k_out, S, ld_S, beta, sc * sc, 0);
    return cudaGetLastError();
}

// ---------------------------------------------------------------- norms
namespace {
// out[r] = sum_f X[r][f]^2 (one warp per row)
__global__ void row_sq_norms_kernel(const float* __restrict__ X, int64_t n, int64_t D, int64_t ld,
                                    float* __restrict__ out) {
    const int64_t r = (int64_t)blockIdx.x * (blockDim.x / 32) + threadIdx.x / 32;
    const int lane = threadIdx.x & 31;
    if (r >= n) return;
    float s = 0.f;
    for (int64_t f = lane; f < D; f += 32) {
        const float v = X[r * ld + f];
        s = fmaf(v, v, s);
    }
    for (int o = 16; o > 0; o >>= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
    if (lane == 0) out[r] = s;
}
// C[q][i] = S[q][i] / sqrt(nq[q] * nt[i])
__global__ void cosine_kernel(float* __restrict__ S, int64_t n_q, int64_t n_t, int64_t ld_S,
                              const float* __restrict__ nq, const float* __restrict__ nt) {
    const int64_t total = n_q * n_t;
    for (int64_t e = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; e < total;
         e += (int64_t)gridDim.x * blockDim.x) {
        const int64_t q = e / n_t, i = e - q * n_t;
        S[q * ld_S + i] = S[q * ld_S + i] / sqrtf(nq[q] * nt[i]);
    }
}
}  // namespace

cudaError_t launch_row_sq_norms(const float* X, int64_t n, int64_t D, int64_t ld, float* out, cudaStream_t s) {
    if (n == 0) return cudaSuccess;
    note_launches(1);
    row_sq_norms_kernel<<<(unsigned)((n + 7) / 8), 256, 0, s>>>(X, n, D, ld, out);
    return cudaGetLastError();
}

cudaError_t launch_cosine(float* S, int64_t n_q, int64_t n_t, int64_t ld_S, const float* nq, const float* nt,
                          cudaStream_t s) {
    if (n_q == 0 || n_t == 0) return cudaSuccess;
    int64_t blocks = (n_q * n_t + 255) / 256;
    if (blocks > 152 * 32) blocks = 152 * 32;
    note_launches(1);
    cosine_kernel<<<(unsigned)blocks, 256, 0, s>>>(S, n_q, n_t, ld_S, nq, nt);
    return cudaGetLastError();
}

// ||DW_i||^2 for i in [0, n) by Eq. 4 with both sides example i (unprojected,
// or on projected factors Y laid out as in launch_project_factors with alpha =
// scale^2).
cudaError_t launch_gram_self(const tda_layer_desc& L, tda_dtype dt, const void* A, const void* B, int64_t n,
                             int64_t d_in, int64_t d_out, float alpha, float* out, cudaStream_t s) {
    if (n == 0) return cudaSuccess;
    note_launches(1);
    if (dt == TDA_BF16)
        gram_kernel<__nv_bfloat16><<<(unsigned)n, kTh, 0, s>>>((const __nv_bfloat16*)A, (const __nv_bfloat16*)B,
                                                               (const __nv_bfloat16*)A, (const __nv_bfloat16*)B, L.T,
                                                               d_in, d_out, out, 0, 0.f, alpha, 1);
    else
        gram_kernel<float><<<(unsigned)n, kTh, 0, s>>>((const float*)A, (const float*)B, (const float*)A,
                                                       (const float*)B, L.T, d_in, d_out, out, 0, 0.f, alpha, 1);
    return cudaGetLastError();
}

cudaError_t launch_materialize_G(const tda_layer_desc& L, tda_dtype dt, const void* A, const void* B, int64_t e0,
                                 int64_t n, float* G, cudaStream_t s) {
    if (n == 0) return cudaSuccess;
    if (dt == TDA_BF16)
        launch_materialize<__nv_bfloat16>(A, B, e0, n, L, G, s);
    else
        launch_materialize<float>(A, B, e0, n, L, G, s);
    return cudaGetLastError();
}

}  // namespace tda
