// k_precond.cu -- damped Fisher preconditioner of the queries.
//
// App. B.3: curvature-based methods fit a curvature matrix over the training
// gradients and precondition the queries layer by layer; App. B.2: damping is
// a multiple of the layer's mean eigenvalue. On projected features phi (D per
// example) the fit is the empirical Fisher F = (1/N) sum_i phi_i phi_i^T, and a
// query q becomes qhat = (F + lambda I)^{-1} q.
//
// State (caller-owned): kPcHeaderDoubles doubles of header, then M (D x D,
// float or double). FIT accumulates M += Phi^T Phi; FACTOR turns M into the
// lower Cholesky factor L of M/n_total + lambda I (blocked right-looking:
// diagonal block, panel triangular solve, trailing update); APPLY solves
// L L^T x = q by blocked forward and backward substitution.
#include <math.h>

#include "tda_internal.cuh"

namespace tda {
namespace {

constexpr int kFT = 64;  // fit tile edge
constexpr int kFK = 32;  // rows per fit chunk
constexpr int kNB = 32;  // Cholesky / substitution block

template <typename TS>
__device__ __forceinline__ TS* mat_of(void* state) {
    return (TS*)((char*)state + kPcHeaderDoubles * sizeof(double));
}
template <typename TS>
__device__ __forceinline__ const TS* mat_of(const void* state) {
    return (const TS*)((const char*)state + kPcHeaderDoubles * sizeof(double));
}

// M[a][b] += sum_n phi[n][a] phi[n][b], 64 x 64 tiles, 256 threads x 4x4.
template <typename TS>
__global__ void __launch_bounds__(256)
pc_fit_kernel(int64_t D, void* state, const float* __restrict__ phi, int64_t n, int64_t ld) {
    __shared__ TS Xa[kFK][kFT + 1];
    __shared__ TS Xb[kFK][kFT + 1];
    TS* M = mat_of<TS>(state);
    const int tid = threadIdx.x, ty = tid / 16, tx = tid % 16;
    const int64_t a0 = (int64_t)blockIdx.y * kFT, b0 = (int64_t)blockIdx.x * kFT;
    TS acc[4][4];
#pragma unroll
    for (int u = 0; u < 4; ++u)
#pragma unroll
        for (int v = 0; v < 4; ++v) acc[u][v] = (TS)0;
    for (int64_t r0 = 0; r0 < n; r0 += kFK) {
        for (int e = tid; e < kFK * kFT; e += 256) {
            const int rr = e / kFT, cc = e % kFT;
            const int64_t r = r0 + rr;
            Xa[rr][cc] = (r < n && a0 + cc < D) ? (TS)phi[r * ld + a0 + cc] : (TS)0;
            Xb[rr][cc] = (r < n && b0 + cc < D) ? (TS)phi[r * ld + b0 + cc] : (TS)0;
        }
        __syncthreads();
#pragma unroll 8
        for (int rr = 0; rr < kFK; ++rr) {
            TS x[4], y[4];
#pragma unroll
            for (int u = 0; u < 4; ++u) x[u] = Xa[rr][ty * 4 + u];
#pragma unroll
            for (int v = 0; v < 4; ++v) y[v] = Xb[rr][tx * 4 + v];
#pragma unroll
            for (int u = 0; u < 4; ++u)
#pragma unroll
                for (int v = 0; v < 4; ++v) acc[u][v] += x[u] * y[v];
        }
        __syncthreads();
    }
#pragma unroll
    for (int u = 0; u < 4; ++u)
#pragma unroll
        for (int v = 0; v < 4; ++v) {
            const int64_t a = a0 + ty * 4 + u, b = b0 + tx * 4 + v;
            if (a < D && b < D) M[a * D + b] += acc[u][v];
        }
}

// Header: trace -> mean eigenvalue of F = M/n_total, and lambda.
template <typename TS>
__global__ void pc_prepare_kernel(int64_t D, void* state, int64_t n_total, double lambda_abs,
                                  double lambda_rel) {
    __shared__ double part[256];
    const TS* M = mat_of<TS>((const void*)state);
    double s = 0.0;
    for (int64_t a = threadIdx.x; a < D; a += blockDim.x) s += (double)M[a * D + a];
    part[threadIdx.x] = s;
    __syncthreads();
    for (int w = blockDim.x / 2; w > 0; w >>= 1) {
        if ((int)threadIdx.x < w) part[threadIdx.x] += part[threadIdx.x + w];
        __syncthreads();
    }
    if (threadIdx.x == 0) {
        double* h = (double*)state;
        const double mean_eig = part[0] / (double)n_total / (double)D;
        h[kPcLambda] = lambda_abs + lambda_rel * mean_eig;
        h[kPcMeanEig] = mean_eig;
        h[kPcFailedPivot] = 0.0;
        h[kPcNTotal] = (double)n_total;
    }
}

// M <- M / n_total + lambda I
template <typename TS>
__global__ void pc_scale_kernel(int64_t D, void* state) {
    const double* h = (const double*)state;
    TS* M = mat_of<TS>(state);
    const TS inv = (TS)(1.0 / h[kPcNTotal]);
    const TS lam = (TS)h[kPcLambda];
    const int64_t total = D * D;
    for (int64_t e = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; e < total;
         e += (int64_t)gridDim.x * blockDim.x) {
        const int64_t a = e / D, b = e - a * D;
        TS v = M[e] * inv;
        if (a == b) v += lam;
        M[e] = v;
    }
}

// Factor the nb x nb diagonal block at k0 in shared memory (unblocked,
// right-looking). A non-positive pivot records its 1-based global index.
template <typename TS>
__global__ void __launch_bounds__(256) pc_chol_diag_kernel(int64_t D, void* state, int64_t k0) {
    __shared__ TS Ls[kNB][kNB + 1];
    TS* M = mat_of<TS>(state);
    double* h = (double*)state;
    const int nb = (int)((D - k0) < kNB ? (D - k0) : kNB);
    for (int e = threadIdx.x; e < nb * nb; e += blockDim.x) {
        const int i = e / nb, j = e % nb;
        Ls[i][j] = M[(k0 + i) * D + k0 + j];
    }
    __syncthreads();
    for (int j = 0; j < nb; ++j) {
        if (threadIdx.x == 0) {
            const TS p = Ls[j][j];
            if (!(p > (TS)0)) {
                if (h[kPcFailedPivot] == 0.0) h[kPcFailedPivot] = (double)(k0 + j + 1);
                Ls[j][j] = (TS)NAN;
            } else {
                Ls[j][j] = sqrt(p);
            }
        }
        __syncthreads();
        const TS piv = Ls[j][j];
        for (int i = j + 1 + threadIdx.x; i < nb; i += blockDim.x) Ls[i][j] /= piv;
        __syncthreads();
        for (int e = threadIdx.x; e < nb * nb; e += blockDim.x) {
            const int i = e / nb, c = e % nb;
            if (i > j && c > j && c <= i) Ls[i][c] -= Ls[i][j] * Ls[c][j];
        }
        __syncthreads();
    }
    for (int e = threadIdx.x; e < nb * nb; e += blockDim.x) {
        const int i = e / nb, j = e % nb;
        M[(k0 + i) * D + k0 + j] = (j <= i) ? Ls[i][j] : (TS)0;
    }
}

// Panel: rows i >= k0+nb solve x L_kk^T = a for their nb entries of block column k0.
template <typename TS>
__global__ void __launch_bounds__(128) pc_chol_panel_kernel(int64_t D, void* state, int64_t k0) {
    __shared__ TS Lk[kNB][kNB + 1];
    TS* M = mat_of<TS>(state);
    const int nb = (int)((D - k0) < kNB ? (D - k0) : kNB);
    for (int e = threadIdx.x; e < nb * nb; e += blockDim.x) {
        const int i = e / nb, j = e % nb;
        Lk[i][j] = M[(k0 + i) * D + k0 + j];
    }
    __syncthreads();
    const int64_t i = k0 + nb + (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    if (i >= D) return;
    TS x[kNB];
    for (int j = 0; j < nb; ++j) {
        TS s = M[i * D + k0 + j];
        for (int m = 0; m < j; ++m) s -= x[m] * Lk[j][m];
        x[j] = s / Lk[j][j];
    }
    for (int j = 0; j < nb; ++j) M[i * D + k0 + j] = x[j];
}

// Trailing update of the lower triangle: M[i][j] -= sum_m L[i][m] L[j][m] over
// the panel columns m in [k0, k0+nb), for i >= j >= k0+nb. 64x64 tiles.
template <typename TS>
__global__ void __launch_bounds__(256) pc_chol_update_kernel(int64_t D, void* state, int64_t k0) {
    if (blockIdx.x > blockIdx.y) return;  // strictly-upper tile
    __shared__ TS Pi[kNB][kFT + 1];
    __shared__ TS Pj[kNB][kFT + 1];
    TS* M = mat_of<TS>(state);
    const int nb = (int)((D - k0) < kNB ? (D - k0) : kNB);
    const int64_t s0 = k0 + nb;
    const int64_t i0 = s0 + (int64_t)blockIdx.y * kFT, j0 = s0 + (int64_t)blockIdx.x * kFT;
    const int tid = threadIdx.x, ty = tid / 16, tx = tid % 16;
    for (int e = tid; e < kNB * kFT; e += 256) {
        const int r = e / kNB, m = e % kNB;
        Pi[m][r] = (i0 + r < D && m < nb) ? M[(i0 + r) * D + k0 + m] : (TS)0;
        Pj[m][r] = (j0 + r < D && m < nb) ? M[(j0 + r) * D + k0 + m] : (TS)0;
    }
    __syncthreads();
    TS acc[4][4];
#pragma unroll
    for (int u = 0; u < 4; ++u)
#pragma unroll
        for (int v = 0; v < 4; ++v) acc[u][v] = (TS)0;
    for (int m = 0; m < kNB; ++m) {
#pragma unroll
        for (int u = 0; u < 4; ++u)
#pragma unroll
            for (int v = 0; v < 4; ++v) acc[u][v] += Pi[m][ty * 4 + u] * Pj[m][tx * 4 + v];
    }
#pragma unroll
    for (int u = 0; u < 4; ++u)
#pragma unroll
        for (int v = 0; v < 4; ++v) {
            const int64_t i = i0 + ty * 4 + u, j = j0 + tx * 4 + v;
            if (i < D && j < D && j <= i) M[i * D + j] -= acc[u][v];
        }
}

// One CTA per query row: forward (L y = q) then backward (L^T x = y)
// substitution in blocks of kNB rows; y and x live in shared memory.
template <typename TS>
__global__ void __launch_bounds__(256)
pc_apply_kernel(int64_t D, const void* state, const float* __restrict__ q, int64_t ld_q,
                TS* __restrict__ out, int64_t ld_out) {
    extern __shared__ __align__(16) unsigned char smem_raw[];
    TS* y = (TS*)smem_raw;             // D entries
    __shared__ TS part[8][kNB];        // per-warp partial sums
    __shared__ TS r[kNB];
    const TS* L = mat_of<TS>(state);
    const double* h = (const double*)state;
    const int64_t row = blockIdx.x;
    const float* qr = q + row * ld_q;
    TS* xo = out + row * ld_out;
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    if (h[kPcFailedPivot] != 0.0) {
        for (int64_t i = tid; i < D; i += blockDim.x) xo[i] = (TS)NAN;
        return;
    }
    // forward: y[i] = (q[i] - sum_{m<i} L[i][m] y[m]) / L[i][i]
    for (int64_t b0 = 0; b0 < D; b0 += kNB) {
        const int nb = (int)((D - b0) < kNB ? (D - b0) : kNB);
        // r[ii] = q[b0+ii] - sum_{m < b0} L[b0+ii][m] y[m]; warps split rows
        for (int ii = warp; ii < nb; ii += 8) {
            TS s = (TS)0;
            for (int64_t m = lane; m < b0; m += 32) s += L[(b0 + ii) * D + m] * y[m];
            for (int o = 16; o > 0; o >>= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
            if (lane == 0) r[ii] = (TS)qr[b0 + ii] - s;
        }
        __syncthreads();
        if (warp == 0) {
            for (int ii = 0; ii < nb; ++ii) {
                TS s = (lane < ii) ? L[(b0 + ii) * D + b0 + lane] * y[b0 + lane] : (TS)0;
                for (int o = 16; o > 0; o >>= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
                if (lane == 0) y[b0 + ii] = (r[ii] - s) / L[(b0 + ii) * D + b0 + ii];
                __syncwarp();
            }
        }
        __syncthreads();
    }
    // backward: x[i] = (y[i] - sum_{m>i} L[m][i] x[m]) / L[i][i]; x overwrites y
    const int64_t nblk = (D + kNB - 1) / kNB;
    for (int64_t bi = nblk - 1; bi >= 0; --bi) {
        const int64_t b0 = bi * kNB;
        const int nb = (int)((D - b0) < kNB ? (D - b0) : kNB);
        const int64_t e0 = b0 + nb;
        // lane = column ii of the block, warps stride over solved rows m >= e0
        TS s = (TS)0;
        if (lane < nb)
            for (int64_t m = e0 + warp; m < D; m += 8) s += L[m * D + b0 + lane] * y[m];
        part[warp][lane] = s;
        __syncthreads();
        if (warp == 0) {
            TS t = (TS)0;
            for (int w = 0; w < 8; ++w) t += part[w][lane];
            if (lane < nb) r[lane] = y[b0 + lane] - t;
            __syncwarp();
            for (int ii = nb - 1; ii >= 0; --ii) {
                TS u = (lane > ii && lane < nb) ? L[(b0 + lane) * D + b0 + ii] * y[b0 + lane] : (TS)0;
                for (int o = 16; o > 0; o >>= 1) u += __shfl_xor_sync(0xffffffffu, u, o);
                if (lane == 0) y[b0 + ii] = (r[ii] - u) / L[(b0 + ii) * D + b0 + ii];
                __syncwarp();
            }
        }
        __syncthreads();
    }
    for (int64_t i = tid; i < D; i += blockDim.x) xo[i] = y[i];
}

template <typename TS>
cudaError_t factor_impl(int64_t D, void* state, int64_t n_total, double la, double lr,
                        cudaStream_t s) {
    note_launches(2);
    pc_prepare_kernel<TS><<<1, 256, 0, s>>>(D, state, n_total, la, lr);
    int64_t blocks = (D * D + 255) / 256;
    if (blocks > 152 * 32) blocks = 152 * 32;
    pc_scale_kernel<TS><<<(unsigned)blocks, 256, 0, s>>>(D, state);
    for (int64_t k0 = 0; k0 < D; k0 += kNB) {
        note_launches(1);
        pc_chol_diag_kernel<TS><<<1, 256, 0, s>>>(D, state, k0);
        const int64_t rest = D - k0 - kNB;
        if (rest > 0) {
            note_launches(2);
            pc_chol_panel_kernel<TS><<<(unsigned)((rest + 127) / 128), 128, 0, s>>>(D, state, k0);
            const unsigned t = (unsigned)((rest + kFT - 1) / kFT);
            pc_chol_update_kernel<TS><<<dim3(t, t), 256, 0, s>>>(D, state, k0);
        }
    }
    return cudaGetLastError();
}

}  // namespace

cudaError_t launch_pc_fit(int64_t D, tda_dtype sdt, void* state, const float* phi, int64_t n,
                          int64_t ld, cudaStream_t s) {
    if (n == 0) return cudaSuccess;
    const unsigned t = (unsigned)((D + kFT - 1) / kFT);
    note_launches(1);
    if (sdt == TDA_F64)
        pc_fit_kernel<double><<<dim3(t, t), 256, 0, s>>>(D, state, phi, n, ld);
    else
        pc_fit_kernel<float><<<dim3(t, t), 256, 0, s>>>(D, state, phi, n, ld);
    return cudaGetLastError();
}

cudaError_t launch_pc_factor(int64_t D, tda_dtype sdt, void* state, int64_t n_total,
                             double lambda_abs, double lambda_rel, cudaStream_t s) {
    if (sdt == TDA_F64) return factor_impl<double>(D, state, n_total, lambda_abs, lambda_rel, s);
    return factor_impl<float>(D, state, n_total, lambda_abs, lambda_rel, s);
}

cudaError_t launch_pc_apply(int64_t D, tda_dtype sdt, const void* state, const float* q,
                            int64_t n_q, int64_t ld_q, void* qhat, int64_t ld_qhat,
                            cudaStream_t s) {
    if (n_q == 0) return cudaSuccess;
    const size_t el = sdt == TDA_F64 ? sizeof(double) : sizeof(float);
    const size_t smem = (size_t)D * el;
    cudaError_t e;
    note_launches(1);
    if (sdt == TDA_F64) {
        e = cudaFuncSetAttribute(pc_apply_kernel<double>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 (int)smem);
        if (e != cudaSuccess) return e;
        pc_apply_kernel<double><<<(unsigned)n_q, 256, smem, s>>>(D, state, q, ld_q, (double*)qhat,
                                                                  ld_qhat);
    } else {
        e = cudaFuncSetAttribute(pc_apply_kernel<float>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 (int)smem);
        if (e != cudaSuccess) return e;
        pc_apply_kernel<float><<<(unsigned)n_q, 256, smem, s>>>(D, state, q, ld_q, (float*)qhat,
                                                                 ld_qhat);
    }
    return cudaGetLastError();
}

}  // namespace tda
