// k_precond.cu -- damped Fisher preconditioner of the queries, for a batch of
// layers with the same feature count D.
//
// App. B.3: curvature-based methods fit a curvature matrix over the training
// gradients and precondition the queries layer by layer; App. B.2: damping is
// a multiple of the layer's mean eigenvalue. On projected features phi (D per
// example and layer) the fit is the empirical Fisher F = (1/N) sum_i phi_i
// phi_i^T, and a query q becomes qhat = (F + lambda I)^{-1} q.
//
// Per-layer state (caller-owned, tda_precondition_state_bytes each, layers
// back to back): 64-byte header | M (D x D) | Dinv (ceil(D/32) blocks of
// 32 x 32), elements float or double. After FACTOR, M holds L strictly below
// its 32 x 32 diagonal blocks; each diagonal block of L is held as its inverse
// in Dinv.
//   FIT     M += Phi^T Phi (lower 128x128 tiles; register-blocked SYRK)
//   FACTOR  M <- L, L L^T = M/n_total + lambda I: right-looking Cholesky in
//           32-column steps; each step factors the diagonal block inside every
//           panel CTA (so it needs no launch of its own), solves the panel, then
//           updates the trailing lower triangle. The inverse of every diagonal
//           block is kept in Dinv.
//   APPLY   forward and backward block substitution; with Dinv each 32-row
//           block step is a small matrix product instead of a serial chain.
// Every launch covers all layers of the call (grid z or y = layer).
//
// Blocked path (fp32 state, D a multiple of 128 and at least 2048): the same
// right-looking Cholesky in 256-column panels of two 128-column halves. Per
// half: the 128 x 128 diagonal block is factored in shared memory (column by
// column, left-looking; Dinv of its four 32 x 32 blocks) and the rows below
// it are solved against it (x L_BB^T = a); the second half's columns first take
// the first half's update. The trailing lower triangle then takes the rank-256
// update M -= P P^T on the tensor cores (3xTF32, launch_gemm_nt_tc). After the
// last panel, L^T is copied into M's upper triangle. APPLY then solves the
// query rows block by block: a 128-wide triangular solve per panel, and the
// rest of every row updated by a tensor-core product with L's panel (forward)
// or with L^T's panel from the upper triangle (backward).
#include <math.h>

#include "tda_internal.cuh"

namespace tda {
namespace {

constexpr int kNB = 32;  // Cholesky / substitution block

template <typename TS>
struct St {
    char* base;
    int64_t D;
    size_t bytes;
    __device__ __forceinline__ double* header(int l) const { return (double*)(base + (size_t)l * bytes); }
    __device__ __forceinline__ TS* M(int l) const { return (TS*)(base + (size_t)l * bytes + 64); }
    __device__ __forceinline__ TS* Dinv(int l) const { return M(l) + D * D; }
};

template <typename TS>
St<TS> state_of(void* state, int64_t D) {
    St<TS> s;
    s.base = (char*)state;
    s.D = D;
    s.bytes = tda_precondition_state_bytes(D, sizeof(TS) == 8 ? TDA_F64 : TDA_F32);
    return s;
}

// ---------------------------------------------------------------- FIT (fp32)
// Tile 128 x 128 of M for rows a0.., cols b0.. (b-tile <= a-tile), K = rows of
// Phi in chunks of 16. Thread (ty, tx) of 16 x 16 owns rows {ty*4+u, 64+ty*4+u}
// and columns {tx*4+v, 64+tx*4+v}: 8 x 8 accumulators, float4 shared reads.
constexpr int kFT = 128, kFK = 16;

__global__ void __launch_bounds__(256, 2)
fit_f32_kernel(St<float> st, const float* __restrict__ phi, int64_t n, int64_t ld) {
    if (blockIdx.x > blockIdx.y) return;  // upper tile: M is used through its lower triangle
    __shared__ __align__(16) float Xa[kFK][kFT];
    __shared__ __align__(16) float Xb[kFK][kFT];
    const int l = blockIdx.z;
    const int64_t D = st.D;
    const float* ph = phi + (int64_t)l * D;
    const int64_t a0 = (int64_t)blockIdx.y * kFT, b0 = (int64_t)blockIdx.x * kFT;
    const int tid = threadIdx.x, ty = tid >> 4, tx = tid & 15;
    float acc[8][8];
#pragma unroll
    for (int u = 0; u < 8; ++u)
#pragma unroll
        for (int v = 0; v < 8; ++v) acc[u][v] = 0.f;
    const bool vec = ((ld & 3) == 0) && ((D & 3) == 0) && (((uintptr_t)ph & 15) == 0);
    for (int64_t r0 = 0; r0 < n; r0 += kFK) {
        // 16 rows x 128 columns per operand: 512 float4 each, 2 per thread
#pragma unroll
        for (int h = 0; h < 2; ++h) {
            const int e = tid + h * 256;
            const int rr = e >> 5, c4 = (e & 31) * 4;
            const int64_t r = r0 + rr;
            float4 va = make_float4(0.f, 0.f, 0.f, 0.f), vb = va;
            if (r < n) {
                const float* row = ph + r * ld;
                if (vec && a0 + c4 + 3 < D) {
                    va = *reinterpret_cast<const float4*>(row + a0 + c4);
                } else {
                    float t[4];
                    for (int i = 0; i < 4; ++i) t[i] = (a0 + c4 + i < D) ? row[a0 + c4 + i] : 0.f;
                    va = make_float4(t[0], t[1], t[2], t[3]);
                }
                if (vec && b0 + c4 + 3 < D) {
                    vb = *reinterpret_cast<const float4*>(row + b0 + c4);
                } else {
                    float t[4];
                    for (int i = 0; i < 4; ++i) t[i] = (b0 + c4 + i < D) ? row[b0 + c4 + i] : 0.f;
                    vb = make_float4(t[0], t[1], t[2], t[3]);
                }
            }
            *reinterpret_cast<float4*>(&Xa[rr][c4]) = va;
            *reinterpret_cast<float4*>(&Xb[rr][c4]) = vb;
        }
        __syncthreads();
#pragma unroll
        for (int k = 0; k < kFK; ++k) {
            const float4 x0 = *reinterpret_cast<const float4*>(&Xa[k][ty * 4]);
            const float4 x1 = *reinterpret_cast<const float4*>(&Xa[k][64 + ty * 4]);
            const float4 y0 = *reinterpret_cast<const float4*>(&Xb[k][tx * 4]);
            const float4 y1 = *reinterpret_cast<const float4*>(&Xb[k][64 + tx * 4]);
            const float x[8] = {x0.x, x0.y, x0.z, x0.w, x1.x, x1.y, x1.z, x1.w};
            const float y[8] = {y0.x, y0.y, y0.z, y0.w, y1.x, y1.y, y1.z, y1.w};
#pragma unroll
            for (int u = 0; u < 8; ++u)
#pragma unroll
                for (int v = 0; v < 8; ++v) acc[u][v] = fmaf(x[u], y[v], acc[u][v]);
        }
        __syncthreads();
    }
    float* M = st.M(l);
#pragma unroll
    for (int u = 0; u < 8; ++u) {
        const int64_t a = a0 + (u < 4 ? ty * 4 + u : 64 + ty * 4 + (u - 4));
        if (a >= D) continue;
#pragma unroll
        for (int v = 0; v < 8; ++v) {
            const int64_t b = b0 + (v < 4 ? tx * 4 + v : 64 + tx * 4 + (v - 4));
            if (b < D) M[a * D + b] += acc[u][v];
        }
    }
}

// ---------------------------------------------------------------- FIT (fp64)
__global__ void __launch_bounds__(256)
fit_f64_kernel(St<double> st, const float* __restrict__ phi, int64_t n, int64_t ld) {
    if (blockIdx.x > blockIdx.y) return;
    constexpr int T = 64, K = 32;
    __shared__ double Xa[K][T + 1];
    __shared__ double Xb[K][T + 1];
    const int l = blockIdx.z;
    const int64_t D = st.D;
    const float* ph = phi + (int64_t)l * D;
    const int tid = threadIdx.x, ty = tid / 16, tx = tid % 16;
    const int64_t a0 = (int64_t)blockIdx.y * T, b0 = (int64_t)blockIdx.x * T;
    double acc[4][4] = {};
    for (int64_t r0 = 0; r0 < n; r0 += K) {
        for (int e = tid; e < K * T; e += 256) {
            const int rr = e / T, cc = e % T;
            const int64_t r = r0 + rr;
            Xa[rr][cc] = (r < n && a0 + cc < D) ? (double)ph[r * ld + a0 + cc] : 0.0;
            Xb[rr][cc] = (r < n && b0 + cc < D) ? (double)ph[r * ld + b0 + cc] : 0.0;
        }
        __syncthreads();
        for (int rr = 0; rr < K; ++rr)
#pragma unroll
            for (int u = 0; u < 4; ++u)
#pragma unroll
                for (int v = 0; v < 4; ++v) acc[u][v] += Xa[rr][ty * 4 + u] * Xb[rr][tx * 4 + v];
        __syncthreads();
    }
    double* M = st.M(l);
    for (int u = 0; u < 4; ++u)
        for (int v = 0; v < 4; ++v) {
            const int64_t a = a0 + ty * 4 + u, b = b0 + tx * 4 + v;
            if (a < D && b < D) M[a * D + b] += acc[u][v];
        }
}

// ---------------------------------------------------------------- FACTOR
// Header: mean eigenvalue of F = M/n_total is tr(M)/(n_total D); lambda.
template <typename TS>
__global__ void prepare_kernel(St<TS> st, int64_t n_total, double lambda_abs, double lambda_rel) {
    __shared__ double part[256];
    const int l = blockIdx.x;
    const int64_t D = st.D;
    const TS* M = st.M(l);
    double s = 0.0;
    for (int64_t a = threadIdx.x; a < D; a += blockDim.x) s += (double)M[a * D + a];
    part[threadIdx.x] = s;
    __syncthreads();
    for (int w = blockDim.x / 2; w > 0; w >>= 1) {
        if ((int)threadIdx.x < w) part[threadIdx.x] += part[threadIdx.x + w];
        __syncthreads();
    }
    if (threadIdx.x == 0) {
        double* h = st.header(l);
        const double mean_eig = part[0] / (double)n_total / (double)D;
        h[kPcLambda] = lambda_abs + lambda_rel * mean_eig;
        h[kPcMeanEig] = mean_eig;
        h[kPcFailedPivot] = 0.0;
        h[kPcNTotal] = (double)n_total;
    }
}

// Lower triangle of M <- M / n_total + lambda I.
template <typename TS>
__global__ void scale_kernel(St<TS> st, int n_layers) {
    const int64_t D = st.D, per = D * D;
    for (int64_t e = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; e < per * n_layers;
         e += (int64_t)gridDim.x * blockDim.x) {
        const int l = (int)(e / per);
        const int64_t r = e - (int64_t)l * per, a = r / D, b = r - a * D;
        if (b > a) continue;
        const double* h = st.header(l);
        TS* M = st.M(l);
        TS v = M[r] * (TS)(1.0 / h[kPcNTotal]);
        if (a == b) v += (TS)h[kPcLambda];
        M[r] = v;
    }
}

// One 32-column step at k0, grid (layer, row chunk): every CTA factors the
// diagonal block in shared memory (one warp), then solves x L_kk^T = a for 256
// panel rows. Row chunk 0 also writes L_kk and its inverse (into Dinv).
template <typename TS>
__global__ void __launch_bounds__(256) panel_kernel(St<TS> st, int64_t k0) {
    __shared__ TS Lk[kNB][kNB + 1];
    const int l = blockIdx.x;
    const int64_t D = st.D;
    TS* M = st.M(l);
    const int nb = (int)((D - k0) < kNB ? (D - k0) : kNB);
    const int tid = threadIdx.x, lane = tid & 31;
    for (int e = tid; e < kNB * kNB; e += blockDim.x) {
        const int i = e / kNB, j = e % kNB;
        TS v;
        if (i < nb && j < nb)
            v = (j <= i) ? M[(k0 + i) * D + k0 + j] : (TS)0;
        else
            v = (i == j) ? (TS)1 : (TS)0;  // identity padding of a ragged last block
        Lk[i][j] = v;
    }
    __syncthreads();
    if (tid < 32) {
        // Lane i holds row i of the block in registers; step j broadcasts the
        // pivot and the scaled column j with warp shuffles (right-looking).
        TS r[kNB];
#pragma unroll
        for (int c = 0; c < kNB; ++c) r[c] = Lk[lane][c];
        int bad = -1;
#pragma unroll
        for (int j = 0; j < kNB; ++j) {
            const TS p = __shfl_sync(0xffffffffu, r[j], j);
            const bool ok = p > (TS)0;
            if (!ok && bad < 0) bad = j;
            const TS piv = ok ? sqrt(p) : (TS)NAN;  // sqrtf for a float state
            if (lane == j) r[j] = piv;
            if (lane > j) r[j] /= piv;
#pragma unroll
            for (int c = j + 1; c < kNB; ++c) {
                const TS v = __shfl_sync(0xffffffffu, r[j], c);  // L[c][j]
                if (lane >= c) r[c] -= r[j] * v;
            }
        }
#pragma unroll
        for (int c = 0; c < kNB; ++c) Lk[lane][c] = (c <= lane) ? r[c] : (TS)0;
        if (blockIdx.y == 0 && lane == 0 && bad >= 0 && bad < nb) {
            double* h = st.header(l);
            if (h[kPcFailedPivot] == 0.0) h[kPcFailedPivot] = (double)(k0 + bad + 1);
        }
    }
    __syncthreads();
    // The diagonal block of M is left as it is: other CTAs of this launch read
    // it, and later steps use the block only through its inverse in Dinv.
    if (blockIdx.y == 0) {
        // inverse of the (padded) diagonal block: lane c solves L X[:, c] = e_c
        if (tid < 32) {
            TS* Di = st.Dinv(l) + (k0 / kNB) * (kNB * kNB);
            const int c = lane;
            TS x[kNB];
#pragma unroll
            for (int i = 0; i < kNB; ++i) {
                TS s = (i == c) ? (TS)1 : (TS)0;
#pragma unroll
                for (int m = 0; m < i; ++m) s -= Lk[i][m] * x[m];
                x[i] = (i < c) ? (TS)0 : s / Lk[i][i];
            }
#pragma unroll
            for (int i = 0; i < kNB; ++i) Di[i * kNB + c] = x[i];
        }
    }
    const int64_t i = k0 + nb + (int64_t)blockIdx.y * blockDim.x + tid;
    if (i >= D) return;
    TS x[kNB];
#pragma unroll
    for (int j = 0; j < kNB; ++j) x[j] = (j < nb) ? M[i * D + k0 + j] : (TS)0;
#pragma unroll
    for (int j = 0; j < kNB; ++j) {
        TS s = x[j];
#pragma unroll
        for (int m = 0; m < j; ++m) s -= x[m] * Lk[j][m];
        x[j] = s / Lk[j][j];
    }
#pragma unroll
    for (int j = 0; j < kNB; ++j)
        if (j < nb) M[i * D + k0 + j] = x[j];
}

// Trailing update of the lower triangle: M[i][j] -= sum_m L[i][m] L[j][m] over
// the panel columns m in [k0, k0+nb), i >= j >= k0+nb. 64x64 tiles, grid z = layer.
template <typename TS>
__global__ void __launch_bounds__(256) update_kernel(St<TS> st, int64_t k0) {
    if (blockIdx.x > blockIdx.y) return;
    constexpr int T = 64;
    __shared__ TS Pi[kNB][T + 1];
    __shared__ TS Pj[kNB][T + 1];
    const int l = blockIdx.z;
    const int64_t D = st.D;
    TS* M = st.M(l);
    const int nb = (int)((D - k0) < kNB ? (D - k0) : kNB);
    const int64_t s0 = k0 + nb;
    const int64_t i0 = s0 + (int64_t)blockIdx.y * T, j0 = s0 + (int64_t)blockIdx.x * T;
    const int tid = threadIdx.x, ty = tid / 16, tx = tid % 16;
    for (int e = tid; e < kNB * T; e += 256) {
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
#pragma unroll 8
    for (int m = 0; m < kNB; ++m) {
        TS a[4], b[4];
#pragma unroll
        for (int u = 0; u < 4; ++u) a[u] = Pi[m][ty * 4 + u];
#pragma unroll
        for (int v = 0; v < 4; ++v) b[v] = Pj[m][tx * 4 + v];
#pragma unroll
        for (int u = 0; u < 4; ++u)
#pragma unroll
            for (int v = 0; v < 4; ++v) acc[u][v] += a[u] * b[v];
    }
#pragma unroll
    for (int u = 0; u < 4; ++u)
#pragma unroll
        for (int v = 0; v < 4; ++v) {
            const int64_t i = i0 + ty * 4 + u, j = j0 + tx * 4 + v;
            if (i < D && j < D && j <= i) M[i * D + j] -= acc[u][v];
        }
}

// ---------------------------------------------------------------- APPLY
// grid (query group, layer). G query rows per CTA; y[G][D] in shared memory.
// Forward, block b:  r = q_b - L_{b,<b} y_<b ;  y_b = Dinv_b r
// Backward, block b: r = y_b - L_{>b,b}^T x_>b ;  x_b = Dinv_b^T r
template <typename TS, int G>
__global__ void __launch_bounds__(256)
apply_kernel(St<TS> st, const float* __restrict__ q, int64_t n_q, int64_t ld_q, TS* __restrict__ out,
             int64_t ld_out) {
    extern __shared__ __align__(16) unsigned char smem_raw[];
    TS* y = (TS*)smem_raw;  // [G][D]
    __shared__ TS part[8][G][kNB];
    __shared__ TS r[G][kNB];
    __shared__ TS Dsm[kNB][kNB + 1];  // inverse of the current diagonal block
    const int l = blockIdx.y;
    const int64_t D = st.D;
    const TS* L = st.M(l);
    const TS* Dv = st.Dinv(l);
    const double* h = st.header(l);
    const int64_t g0 = (int64_t)blockIdx.x * G;
    const int gn = (int)((n_q - g0) < G ? (n_q - g0) : G);
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    if (h[kPcFailedPivot] != 0.0) {
        for (int g = 0; g < gn; ++g)
            for (int64_t i = tid; i < D; i += blockDim.x) out[(g0 + g) * ld_out + (int64_t)l * D + i] = (TS)NAN;
        return;
    }
    const int64_t nblk = (D + kNB - 1) / kNB;
    // forward
    for (int64_t bi = 0; bi < nblk; ++bi) {
        const int64_t b0 = bi * kNB;
        const int nb = (int)((D - b0) < kNB ? (D - b0) : kNB);
        for (int e = tid; e < kNB * kNB; e += blockDim.x) Dsm[e / kNB][e % kNB] = Dv[bi * kNB * kNB + e];
        for (int ii = warp; ii < kNB; ii += 8) {
            TS acc[G];
#pragma unroll
            for (int g = 0; g < G; ++g) acc[g] = (TS)0;
            if (ii < nb)
#pragma unroll 8
                for (int64_t m = lane; m < b0; m += 32) {
                    const TS lv = L[(b0 + ii) * D + m];
#pragma unroll
                    for (int g = 0; g < G; ++g) acc[g] += lv * y[g * D + m];
                }
#pragma unroll
            for (int g = 0; g < G; ++g) {
                TS s = acc[g];
                for (int o = 16; o > 0; o >>= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
                if (lane == 0)
                    r[g][ii] = (ii < nb && g < gn) ? (TS)q[(g0 + g) * ld_q + (int64_t)l * D + b0 + ii] - s : (TS)0;
            }
        }
        __syncthreads();
        for (int e = tid; e < G * kNB; e += blockDim.x) {
            const int g = e / kNB, i = e % kNB;
            TS s = (TS)0;
            for (int j = 0; j <= i; ++j) s += Dsm[i][j] * r[g][j];
            if (i < nb) y[g * D + b0 + i] = s;
        }
        __syncthreads();
    }
    // backward (x overwrites y)
    for (int64_t bi = nblk - 1; bi >= 0; --bi) {
        const int64_t b0 = bi * kNB;
        const int nb = (int)((D - b0) < kNB ? (D - b0) : kNB);
        const int64_t e0 = b0 + nb;
        for (int e = tid; e < kNB * kNB; e += blockDim.x) Dsm[e / kNB][e % kNB] = Dv[bi * kNB * kNB + e];
        TS acc[G];
#pragma unroll
        for (int g = 0; g < G; ++g) acc[g] = (TS)0;
        if (lane < nb)
#pragma unroll 8
            for (int64_t m = e0 + warp; m < D; m += 8) {
                const TS lv = L[m * D + b0 + lane];
#pragma unroll
                for (int g = 0; g < G; ++g) acc[g] += lv * y[g * D + m];
            }
#pragma unroll
        for (int g = 0; g < G; ++g) part[warp][g][lane] = acc[g];
        __syncthreads();
        for (int e = tid; e < G * kNB; e += blockDim.x) {
            const int g = e / kNB, i = e % kNB;
            TS t = (TS)0;
            for (int w = 0; w < 8; ++w) t += part[w][g][i];
            r[g][i] = (i < nb) ? y[g * D + b0 + i] - t : (TS)0;
        }
        __syncthreads();
        for (int e = tid; e < G * kNB; e += blockDim.x) {
            const int g = e / kNB, i = e % kNB;
            TS s = (TS)0;
            for (int j = i; j < kNB; ++j) s += Dsm[j][i] * r[g][j];
            if (i < nb) y[g * D + b0 + i] = s;
        }
        __syncthreads();
    }
    for (int g = 0; g < gn; ++g)
        for (int64_t i = tid; i < D; i += blockDim.x) out[(g0 + g) * ld_out + (int64_t)l * D + i] = y[g * D + i];
}

// ---------------------------------------------------------------- FACTOR in one launch (fp32)
// The same right-looking Cholesky in 32-column steps, with one thread-block
// cluster of CS CTAs per layer instead of two launches per step: every CTA
// factors the diagonal block, the CTAs share the panel rows and the trailing
// 64 x 64 tiles, and cluster barriers separate the phases. M is read through
// L2 (ld.global.cg): other CTAs of the cluster wrote it. Each step does the
// arithmetic of prepare/scale/panel/update_kernel in the same order; the
// factored diagonal blocks are kept in M's diagonal blocks and inverted into
// Dinv after the last step, one warp per block.
__device__ __forceinline__ uint32_t cluster_ctarank() {
    uint32_t r;
    asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
    return r;
}
// release / acquire at cluster scope order every earlier global and shared access of
// the arriving threads before every later access of the waiting ones: the data the CTAs
// exchange through M (read back with ld.global.cg) needs no separate device-wide fence
__device__ __forceinline__ void cluster_barrier() {
    asm volatile("barrier.cluster.arrive.release.aligned;\n barrier.cluster.wait.acquire.aligned;" ::: "memory");
}

// Cholesky of a 32 x 32 block by one warp. Lane i holds row i of the block
// in registers, shifted so that r[0] is always the column being eliminated:
// the step loop stays rolled (compact code; every array index is static).
// Column j of L goes to row j of LkT (LkT[j][i] = L[i][j], zero above the
// diagonal), 1 / L_jj to dinv[j]. Returns the first non-positive pivot's
// column or -1.
__device__ __forceinline__ int warp_cholesky32(const float (*A)[kNB + 1], float (*LkT)[2 * kNB + 1],
                                               float* dinv, int lane) {
    float r[kNB];
#pragma unroll
    for (int c = 0; c < kNB; ++c) r[c] = A[lane][c];
    int bad = -1;
#pragma unroll 1
    for (int j = 0; j < kNB; ++j) {
        const float p = __shfl_sync(0xffffffffu, r[0], j);
        const bool ok = p > 0.f;
        if (!ok && bad < 0) bad = j;
        // L_jj = p * rsqrt(p) and 1 / L_jj = rsqrt(p): one special-function op on the
        // serial path instead of a rounded square root and a division
        const float inv = ok ? rsqrtf(p) : NAN;
        const float piv = p * inv;
        if (lane == j) r[0] = piv;
        else if (lane > j) r[0] *= inv;
        LkT[j][lane] = (lane >= j) ? r[0] : 0.f;
        if (lane == 0) dinv[j] = inv;
        // A[i][j + idx] -= L[i][j] L[j + idx][j] below the diagonal
#pragma unroll
        for (int idx = 1; idx < kNB; ++idx) {
            const float v = __shfl_sync(0xffffffffu, r[0], (j + idx) & (kNB - 1));
            if (lane >= j + idx) r[idx] -= r[0] * v;
        }
#pragma unroll
        for (int idx = 0; idx < kNB - 1; ++idx) r[idx] = r[idx + 1];
        r[kNB - 1] = 0.f;
    }
    return bad;
}

// Queries solved inside the factorisation (FACTOR_APPLY): the query rows ride
// along as extra rows below M -- solved against each diagonal block and updated
// by each panel, which is the forward substitution L y = q -- and a second sweep
// from the last block to the first does the backward substitution L^T x = y.
// CTA r of the cluster keeps the query columns of the 64-wide tiles t with
// t % CS == r in shared memory for the whole call; the owner of a block's
// columns solves that block for all queries and the others read the result
// through distributed shared memory (two buffers, alternating by step).
constexpr int kQT = 64, kQP = kQT + 4;  // query column tile and its padded row
constexpr int kXS = kNB + 4;            // row stride of a solved block: 16-byte rows
// 16 bytes of CTA `rank`'s shared memory at the address of p in this CTA
__device__ __forceinline__ float4 ld_peer4(const float* p, uint32_t rank) {
    uint32_t a = (uint32_t)__cvta_generic_to_shared(p), r;
    asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(r) : "r"(a), "r"(rank));
    float4 v;
    asm volatile("ld.shared::cluster.v4.f32 {%0, %1, %2, %3}, [%4];" : "=f"(v.x), "=f"(v.y), "=f"(v.z), "=f"(v.w)
                 : "r"(r));
    return v;
}
// this CTA's copy of the solved block [n_q][kNB] (stride kXS) that CTA `rank` holds at Xo
__device__ __forceinline__ void copy_peer_block(float* XL, const float* Xo, int64_t n_q, uint32_t rank, int tid) {
    const int64_t n4 = n_q * (kNB / 4);
    for (int64_t e0 = tid; e0 < n4; e0 += 4 * 256) {
        float4 v[4];
#pragma unroll
        for (int u = 0; u < 4; ++u) {  // four loads in flight before the first store
            const int64_t e = e0 + u * 256;
            if (e < n4) v[u] = ld_peer4(Xo + (e / (kNB / 4)) * kXS + (e % (kNB / 4)) * 4, rank);
        }
#pragma unroll
        for (int u = 0; u < 4; ++u) {
            const int64_t e = e0 + u * 256;
            if (e < n4) *reinterpret_cast<float4*>(XL + (e / (kNB / 4)) * kXS + (e % (kNB / 4)) * 4) = v[u];
        }
    }
}
__host__ __device__ inline int64_t query_tiles_per_cta(int64_t D, int cs) {
    return ((D + kQT - 1) / kQT + cs - 1) / cs;
}
__host__ __device__ inline size_t solve_smem_bytes(int64_t D, int64_t n_q, int cs) {
    return sizeof(float) * ((size_t)query_tiles_per_cta(D, cs) * n_q * kQP + 3 * (size_t)n_q * kXS);
}
struct QArgs {
    const float* q;   // layer 0's column 0 of query row 0
    float* qhat;
    int64_t n_q, ld_q, ld_qhat;
};

template <int CS, bool SOLVE>
__global__ void __launch_bounds__(256, 1) factor_cluster_kernel(St<float> st, int64_t n_total, double lambda_abs,
                                                              double lambda_rel, QArgs qa) {
    __shared__ float Lk[kNB][kNB + 1];        // the diagonal block before factoring
    __shared__ float LkT[kNB][2 * kNB + 1];   // L transposed; columns 32..63 stay zero
    __shared__ float dinv[kNB];               // 1 / L_jj of the current block
    __shared__ double part[256];
    constexpr int T = 64;
    __shared__ __align__(16) float Pi[kNB][T + 4];  // 16-byte rows: the products read float4
    __shared__ __align__(16) float Pj[kNB][T + 4];
    const int rank = (int)cluster_ctarank();
    const int l = blockIdx.x / CS;
    const int64_t D = st.D;
    float* M = st.M(l);
    double* h = st.header(l);
    const int tid = threadIdx.x, lane = tid & 31, ty = tid / 16, tx = tid % 16;
    const int64_t n_q = SOLVE ? qa.n_q : 0;
    extern __shared__ __align__(16) float qsm[];
    const int64_t nown = SOLVE ? query_tiles_per_cta(D, CS) : 0;
    float* Qs = qsm;                                 // [nown][n_q][kQP]: owned query column tiles
    float* XB = Qs + nown * n_q * kQP;               // [2][n_q][kXS]: a solved block, for the others
    float* XL = XB + 2 * n_q * kXS;                  // [n_q][kXS]: the owner's block, copied here
    for (int e = tid; e < kNB * (2 * kNB + 1); e += blockDim.x) (&LkT[0][0])[e] = 0.f;
    // damping from the mean eigenvalue tr(M)/(n_total D), summed like prepare_kernel
    double s = 0.0;
    for (int64_t a = tid; a < D; a += blockDim.x) s += (double)__ldcg(M + a * D + a);
    part[tid] = s;
    __syncthreads();
    for (int w = blockDim.x / 2; w > 0; w >>= 1) {
        if (tid < w) part[tid] += part[tid + w];
        __syncthreads();
    }
    const double mean_eig = part[0] / (double)n_total / (double)D;
    const double lambda = lambda_abs + lambda_rel * mean_eig;
    if (rank == 0 && tid == 0) {
        h[kPcLambda] = lambda;
        h[kPcMeanEig] = mean_eig;
        h[kPcFailedPivot] = 0.0;
        h[kPcNTotal] = (double)n_total;
    }
    cluster_barrier();  // every CTA has read the diagonal before it is scaled
    {
        const float inv_n = (float)(1.0 / (double)n_total), lam = (float)lambda;
        for (int64_t i = rank; i < D; i += CS)
            for (int64_t j = tid; j <= i; j += blockDim.x) {
                float v = __ldcg(M + i * D + j) * inv_n;
                if (i == j) v += lam;
                M[i * D + j] = v;
            }
        if (SOLVE)
            for (int64_t o = 0; o < nown; ++o) {
                const int64_t c0 = (rank + o * CS) * kQT;
                for (int64_t e = tid; e < n_q * kQT; e += blockDim.x) {
                    const int64_t qi = e / kQT, c = c0 + e % kQT;
                    Qs[(o * n_q + qi) * kQP + e % kQT] = c < D ? qa.q[qi * qa.ld_q + (int64_t)l * D + c] : 0.f;
                }
            }
    }
    cluster_barrier();
    static_assert(CS >= 2, "rank 0 factors the next diagonal block while the others update");
    for (int64_t k0 = 0; k0 < D; k0 += kNB) {
        // ---- diagonal block. The first is factored in registers by warp 0 of every CTA; each
        // later one was factored by rank 0 during the previous step's trailing update (look-
        // ahead: it lies in that update's first tile), which rank 0 keeps in LkT / dinv and the
        // others read back from M's diagonal block and the block's slot of Dinv
        if (k0 == 0) {
            for (int e = tid; e < kNB * kNB; e += blockDim.x) {
                const int i = e / kNB, j = e % kNB;
                Lk[i][j] = (j <= i) ? __ldcg(M + (k0 + i) * D + k0 + j) : 0.f;
            }
            __syncthreads();
            if (tid < 32) {
                const int bad = warp_cholesky32(Lk, LkT, dinv, lane);
                if (rank == 0 && lane == 0 && bad >= 0 && h[kPcFailedPivot] == 0.0) h[kPcFailedPivot] = (double)(k0 + bad + 1);
            }
        } else if (rank != 0) {
            for (int e = tid; e < kNB * kNB; e += blockDim.x) {
                const int i = e / kNB, j = e % kNB;
                LkT[j][i] = (j <= i) ? __ldcg(M + (k0 + i) * D + k0 + j) : 0.f;
            }
            if (tid < kNB) dinv[tid] = __ldcg(st.Dinv(l) + (k0 / kNB) * (kNB * kNB) + tid);
        }
        __syncthreads();
        // ---- panel rows below the block (and the query rows): x L_kk^T = a, every CS-th row
        // to each CTA of the cluster. Column order with the same register shift: once x_j is
        // known it leaves every later entry
        for (int64_t i = k0 + kNB + (int64_t)tid * CS + rank; i < D; i += (int64_t)CS * blockDim.x) {
            float* row = M + i * D + k0;
            float x[kNB];
#pragma unroll
            for (int j = 0; j < kNB; ++j) x[j] = __ldcg(row + j);
#pragma unroll 1
            for (int j = 0; j < kNB; ++j) {
                const float xj = x[0] * dinv[j];
                row[j] = xj;
#pragma unroll
                for (int idx = 1; idx < kNB; ++idx) x[idx] -= xj * LkT[j][j + idx];
#pragma unroll
                for (int idx = 0; idx < kNB - 1; ++idx) x[idx] = x[idx + 1];
                x[kNB - 1] = 0.f;
            }
        }
        const int blk = (int)(k0 / kNB), own = (blk / 2) % CS;  // the block's columns: tile blk / 2
        if (SOLVE && rank == own) {
            // y_b = q~_b L_bb^-T for every query, the same column-order solve as a panel row
            float* Qb = Qs + ((blk / 2) / CS) * n_q * kQP + (blk % 2) * kNB;
            float* Xo = XB + (blk & 1) * n_q * kXS;
            // query rows start at thread 128: the panel rows above keep at most the first
            // ceil((D - 32) / CS) threads busy, so both chains run side by side
            for (int64_t qi = (tid + blockDim.x / 2) % blockDim.x; qi < n_q; qi += blockDim.x) {
                float* row = Qb + qi * kQP;
                float x[kNB];
#pragma unroll
                for (int j = 0; j < kNB; ++j) x[j] = row[j];
#pragma unroll 1
                for (int j = 0; j < kNB; ++j) {
                    const float xj = x[0] * dinv[j];
                    row[j] = xj;
                    Xo[qi * kXS + j] = xj;
#pragma unroll
                    for (int idx = 1; idx < kNB; ++idx) x[idx] -= xj * LkT[j][j + idx];
#pragma unroll
                    for (int idx = 0; idx < kNB - 1; ++idx) x[idx] = x[idx + 1];
                    x[kNB - 1] = 0.f;
                }
            }
        }
        cluster_barrier();
        if (SOLVE && k0 + kNB < D) {
            // q~[:, c] -= y_b L[c][k0..k0+31]^T for the owned columns c >= k0 + 32
            copy_peer_block(XL, XB + (blk & 1) * n_q * kXS, n_q, (uint32_t)own, tid);
            __syncthreads();
            for (int64_t o = 0; o < nown; ++o) {
                const int64_t c0 = (rank + o * CS) * kQT;
                if (c0 + kQT <= k0 + kNB || c0 >= D) continue;
                for (int e = tid; e < kNB * kQT; e += blockDim.x) {
                    const int cc = e / kNB, m = e % kNB;
                    const int64_t c = c0 + cc;
                    Pj[m][cc] = (c >= k0 + kNB && c < D) ? __ldcg(M + c * D + k0 + m) : 0.f;
                }
                __syncthreads();
                for (int64_t q0 = 0; q0 < n_q; q0 += kQT) {
#pragma unroll
                    for (int r = 0; r < 4; ++r) {
                        const int64_t qi = q0 + ty * 4 + r;
                        if (qi >= n_q) break;
                        float acc[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll 8
                        for (int m = 0; m < kNB; ++m) {
                            const float xv = XL[qi * kXS + m];
                            const float4 b4 = *reinterpret_cast<const float4*>(&Pj[m][tx * 4]);
                            acc[0] += xv * b4.x, acc[1] += xv * b4.y, acc[2] += xv * b4.z, acc[3] += xv * b4.w;
                        }
                        float4* dst = reinterpret_cast<float4*>(Qs + (o * n_q + qi) * kQP + tx * 4);
                        float4 v = *dst;
                        v.x -= acc[0], v.y -= acc[1], v.z -= acc[2], v.w -= acc[3];
                        *dst = v;
                    }
                }
                __syncthreads();
            }
        }
        // the factored block goes back into M's diagonal block once every CTA has read the
        // unfactored one (no later step reads that block); the inverses of all diagonal
        // blocks are formed after the last step
        if (k0 == 0 && rank == 0)
            for (int e = tid; e < kNB * kNB; e += blockDim.x) {
                const int i = e / kNB, j = e % kNB;
                if (j <= i) M[(k0 + i) * D + k0 + j] = LkT[j][i];
            }
        // ---- trailing update of the lower triangle (and of the query rows' remaining
        // columns), 64 x 64 tiles shared by the cluster
        const int64_t s0 = k0 + kNB;
        const int64_t rest = D - s0;
        if (rest > 0) {
            const int64_t t = (rest + T - 1) / T, lower = t * (t + 1) / 2;
            const int64_t tiles = lower;
            // tile u: lower-triangle tile (bi, bj), bj <= bi, row-major; then query tiles (qb, bj)
            struct Tile {
                float* rows;  // M or the query rows
                int64_t ld, lim, i0, j0;
                bool tri;     // lower triangle of M: only j <= i
            };
            auto tile_of = [&](int64_t u) {
                Tile tl;
                {
                    // fp32 estimate (fp64 is a slow pipe here), corrected in integers
                    int64_t bi = (int64_t)((sqrtf(8.f * (float)u + 1.f) - 1.f) * 0.5f);
                    while (bi * (bi + 1) / 2 > u) --bi;
                    while ((bi + 1) * (bi + 2) / 2 <= u) ++bi;
                    tl.rows = M, tl.ld = D, tl.lim = D, tl.tri = true;
                    tl.i0 = s0 + bi * T;
                    tl.j0 = s0 + (u - bi * (bi + 1) / 2) * T;
                }
                return tl;
            };
            // software pipeline: while tile u is multiplied, the panel rows and the current
            // values of this CTA's next tile are on their way (each thread: 8 + 8 panel values,
            // row e/32, column e%32, and its 4 x 4 outputs)
            float ra[8], rb[8], mv[4][4];
            auto load_tile = [&](int64_t u) {
                const Tile tl = tile_of(u);
#pragma unroll
                for (int hh = 0; hh < 8; ++hh) {
                    const int e = tid + hh * 256, r = e / kNB, m = e % kNB;
                    ra[hh] = (tl.i0 + r < tl.lim) ? __ldcg(tl.rows + (tl.i0 + r) * tl.ld + k0 + m) : 0.f;
                    rb[hh] = (tl.j0 + r < D) ? __ldcg(M + (tl.j0 + r) * D + k0 + m) : 0.f;
                }
#pragma unroll
                for (int q = 0; q < 4; ++q)
#pragma unroll
                    for (int v = 0; v < 4; ++v) {
                        const int64_t i = tl.i0 + ty * 4 + q, j = tl.j0 + tx * 4 + v;
                        mv[q][v] = (i < tl.lim && j < D && (!tl.tri || j <= i)) ? __ldcg(tl.rows + i * tl.ld + j)
                                                                                 : 0.f;
                    }
            };
            // rank 0 takes tile 0 alone (it holds the next diagonal block, factored right after);
            // ranks 1 .. CS-1 share the others
            const int64_t ustep = rank == 0 ? tiles : CS - 1;
            int64_t u = rank;
            if (u < tiles) load_tile(u);
            for (; u < tiles; u += ustep) {
                const Tile tl = tile_of(u);
#pragma unroll
                for (int hh = 0; hh < 8; ++hh) {
                    const int e = tid + hh * 256, r = e / kNB, m = e % kNB;
                    Pi[m][r] = ra[hh];
                    Pj[m][r] = rb[hh];
                }
                float acc[4][4];
#pragma unroll
                for (int a = 0; a < 4; ++a)
#pragma unroll
                    for (int b = 0; b < 4; ++b) acc[a][b] = mv[a][b];
                __syncthreads();
                if (u + ustep < tiles) load_tile(u + ustep);
#pragma unroll 8
                for (int m = 0; m < kNB; ++m) {
                    const float4 a4 = *reinterpret_cast<const float4*>(&Pi[m][ty * 4]);
                    const float4 b4 = *reinterpret_cast<const float4*>(&Pj[m][tx * 4]);
                    const float a[4] = {a4.x, a4.y, a4.z, a4.w}, b[4] = {b4.x, b4.y, b4.z, b4.w};
#pragma unroll
                    for (int q = 0; q < 4; ++q)
#pragma unroll
                        for (int v = 0; v < 4; ++v) acc[q][v] -= a[q] * b[v];
                }
#pragma unroll
                for (int q = 0; q < 4; ++q)
#pragma unroll
                    for (int v = 0; v < 4; ++v) {
                        const int64_t i = tl.i0 + ty * 4 + q, j = tl.j0 + tx * 4 + v;
                        if (i < tl.lim && j < D && (!tl.tri || j <= i)) tl.rows[i * tl.ld + j] = acc[q][v];
                        // tile 0's top-left 32 x 32: the next diagonal block, updated (D - s0 >= 32)
                        if (u == 0 && ty * 4 + q < kNB && tx * 4 + v < kNB)
                            Lk[ty * 4 + q][tx * 4 + v] = (tx * 4 + v <= ty * 4 + q) ? acc[q][v] : 0.f;
                    }
                __syncthreads();
            }
            if (rank == 0) {
                // look-ahead: factor the next diagonal block now; the others read it after the barrier
                if (tid < 32) {
                    const int bad = warp_cholesky32(Lk, LkT, dinv, lane);
                    if (lane == 0 && bad >= 0 && h[kPcFailedPivot] == 0.0) h[kPcFailedPivot] = (double)(s0 + bad + 1);
                }
                __syncthreads();
                for (int e = tid; e < kNB * kNB; e += blockDim.x) {
                    const int i = e / kNB, j = e % kNB;
                    if (j <= i) M[(s0 + i) * D + s0 + j] = LkT[j][i];
                }
                if (tid < kNB) st.Dinv(l)[(s0 / kNB) * (kNB * kNB) + tid] = dinv[tid];
            }
        }
        cluster_barrier();
    }
    // inverses of the factored diagonal blocks: a CTA stages a block in shared
    // memory and lane c of warp 0 solves L X[:, c] = e_c in column order
    const int nblk = (int)(D / kNB);
    for (int b = rank; b < nblk; b += CS) {
        const float* Lb = M + (int64_t)b * kNB * D + (int64_t)b * kNB;
        for (int e = tid; e < kNB * kNB; e += blockDim.x) {
            const int i = e / kNB, j = e % kNB;
            Lk[i][j] = (j <= i) ? __ldcg(Lb + (int64_t)i * D + j) : 0.f;
        }
        __syncthreads();
        if (tid < kNB) {
            const int c = lane;
            float x[kNB];
#pragma unroll
            for (int i = 0; i < kNB; ++i) x[i] = (i == c) ? 1.f : 0.f;
#pragma unroll
            for (int j = 0; j < kNB; ++j) {
                x[j] = (j < c) ? 0.f : x[j] / Lk[j][j];
#pragma unroll
                for (int i = j + 1; i < kNB; ++i) x[i] -= Lk[i][j] * x[j];
            }
            float* Di = st.Dinv(l) + (int64_t)b * (kNB * kNB);
#pragma unroll
            for (int i = 0; i < kNB; ++i) Di[i * kNB + c] = x[i];
        }
        __syncthreads();
    }
    if constexpr (SOLVE) {
        // ---- backward substitution L^T x = y from the last block: the owner of block b forms
        // x_b = Dinv_b^T y~_b for every query; then each CTA removes x_b L[b0..b0+31][c] from
        // its owned columns c < b0
        cluster_barrier();  // Dinv complete
        const int64_t ldh = qa.ld_qhat;
        float* Qh = qa.qhat + (int64_t)l * D;
        if (__ldcg(&h[kPcFailedPivot]) != 0.0) {
            for (int64_t o = 0; o < nown; ++o) {
                const int64_t c0 = (rank + o * CS) * kQT;
                for (int64_t e = tid; e < n_q * kQT; e += blockDim.x)
                    if (c0 + e % kQT < D) Qh[(e / kQT) * ldh + c0 + e % kQT] = NAN;
            }
            return;
        }
        for (int b = nblk - 1; b >= 0; --b) {
            const int64_t b0 = (int64_t)b * kNB;
            const int own = (b / 2) % CS;
            // L[b0..b0+31][c] of this CTA's first owned tile left of the block does not depend
            // on x_b: staged while the owner solves
            const bool pre = nown > 0 && (int64_t)rank * kQT < b0;
            if (pre)
                for (int e = tid; e < kNB * kQT; e += blockDim.x) {
                    const int m = e / kQT, cc = e % kQT;
                    const int64_t c = (int64_t)rank * kQT + cc;
                    Pj[m][cc] = (c < b0) ? __ldcg(M + (b0 + m) * D + c) : 0.f;
                }
            if (rank == own) {
                const float* Di = st.Dinv(l) + (int64_t)b * (kNB * kNB);
                for (int e = tid; e < kNB * kNB; e += blockDim.x) Lk[e / kNB][e % kNB] = __ldcg(Di + e);
                __syncthreads();
                float* Qb = Qs + ((b / 2) / CS) * n_q * kQP + (b % 2) * kNB;
                float* Xo = XB + (b & 1) * n_q * kXS;
                for (int64_t e = tid; e < n_q * kNB; e += blockDim.x) {
                    const int64_t qi = e / kNB;
                    const int c = (int)(e % kNB);
                    float acc = 0.f;  // Dinv_b is lower triangular: entries above the diagonal are 0
#pragma unroll
                    for (int i = 0; i < kNB; ++i) acc += Lk[i][c] * Qb[qi * kQP + i];
                    Xo[qi * kXS + c] = acc;
                }
                __syncthreads();
                for (int64_t e = tid; e < n_q * kNB; e += blockDim.x)
                    Qb[(e / kNB) * kQP + e % kNB] = Xo[(e / kNB) * kXS + e % kNB];
            }
            cluster_barrier();
            if (b0 == 0) break;
            copy_peer_block(XL, XB + (b & 1) * n_q * kXS, n_q, (uint32_t)own, tid);
            __syncthreads();
            for (int64_t o = 0; o < nown; ++o) {
                const int64_t c0 = (rank + o * CS) * kQT;
                if (c0 >= b0) continue;
                if (o > 0) {
                    for (int e = tid; e < kNB * kQT; e += blockDim.x) {
                        const int m = e / kQT, cc = e % kQT;
                        Pj[m][cc] = (c0 + cc < b0) ? __ldcg(M + (b0 + m) * D + c0 + cc) : 0.f;
                    }
                }
                __syncthreads();
                for (int64_t q0 = 0; q0 < n_q; q0 += kQT) {
#pragma unroll
                    for (int r = 0; r < 4; ++r) {
                        const int64_t qi = q0 + ty * 4 + r;
                        if (qi >= n_q) break;
                        float acc[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll 8
                        for (int m = 0; m < kNB; ++m) {
                            const float xv = XL[qi * kXS + m];
                            const float4 b4 = *reinterpret_cast<const float4*>(&Pj[m][tx * 4]);
                            acc[0] += xv * b4.x, acc[1] += xv * b4.y, acc[2] += xv * b4.z, acc[3] += xv * b4.w;
                        }
                        float4* dst = reinterpret_cast<float4*>(Qs + (o * n_q + qi) * kQP + tx * 4);
                        float4 v = *dst;
                        v.x -= acc[0], v.y -= acc[1], v.z -= acc[2], v.w -= acc[3];
                        *dst = v;
                    }
                }
                __syncthreads();
            }
        }
        // the owned columns now hold x: out to qhat
        for (int64_t o = 0; o < nown; ++o) {
            const int64_t c0 = (rank + o * CS) * kQT;
            for (int64_t e = tid; e < n_q * kQT; e += blockDim.x)
                if (c0 + e % kQT < D) Qh[(e / kQT) * ldh + c0 + e % kQT] = Qs[(o * n_q + e / kQT) * kQP + e % kQT];
        }
        cluster_barrier();  // peers may still read this CTA's exchange buffer
    }
}

template <int CS, bool SOLVE>
cudaError_t factor_cluster(int n_layers, int64_t D, void* state, int64_t n_total, double la, double lr,
                           const QArgs& qa, cudaStream_t s) {
    cudaError_t e = cudaSuccess;
    if (CS > 8)
        e = cudaFuncSetAttribute(factor_cluster_kernel<CS, SOLVE>, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
    if (e != cudaSuccess) return e;
    const size_t smem = SOLVE ? solve_smem_bytes(D, qa.n_q, CS) : 0;
    if (smem > 190 * 1024) return cudaErrorNotSupported;
    if (SOLVE &&
        (e = cudaFuncSetAttribute(factor_cluster_kernel<CS, SOLVE>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                  (int)smem)) != cudaSuccess)
        return e;
    cudaLaunchConfig_t cfg = {};
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = CS;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    cfg.gridDim = dim3((unsigned)(n_layers * CS));
    cfg.blockDim = dim3(256);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = s;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    int max_clusters = 0;
    if (cudaOccupancyMaxActiveClusters(&max_clusters, factor_cluster_kernel<CS, SOLVE>, &cfg) != cudaSuccess ||
        max_clusters < 1) {
        cudaGetLastError();
        return cudaErrorNotSupported;
    }
    note_launches(1);
    e = cudaLaunchKernelEx(&cfg, factor_cluster_kernel<CS, SOLVE>, state_of<float>(state, D), n_total, la, lr, qa);
    if (e != cudaSuccess) return e;
    return cudaGetLastError();
}

template <typename TS>
cudaError_t factor_impl(int n_layers, int64_t D, void* state, int64_t n_total, double la, double lr,
                        cudaStream_t s) {
    if constexpr (sizeof(TS) == 4) {
        // fp32 state, whole 32-column blocks: one launch, a cluster of 16 (else 8) CTAs per layer
        if (D % kNB == 0 && D >= 2 * kNB) {
            const QArgs none{nullptr, nullptr, 0, 0, 0};
            cudaError_t e = factor_cluster<16, false>(n_layers, D, state, n_total, la, lr, none, s);
            if (e == cudaErrorNotSupported) e = factor_cluster<8, false>(n_layers, D, state, n_total, la, lr, none, s);
            if (e != cudaErrorNotSupported) return e;
        }
    }
    St<TS> st = state_of<TS>(state, D);
    note_launches(2);
    prepare_kernel<TS><<<n_layers, 256, 0, s>>>(st, n_total, la, lr);
    int64_t blocks = (D * D * n_layers + 255) / 256;
    if (blocks > 152 * 16) blocks = 152 * 16;
    scale_kernel<TS><<<(unsigned)blocks, 256, 0, s>>>(st, n_layers);
    for (int64_t k0 = 0; k0 < D; k0 += kNB) {
        const int64_t rest = D - k0 - kNB;
        const unsigned chunks = (unsigned)(rest > 0 ? (rest + 255) / 256 : 1);
        note_launches(1);
        panel_kernel<TS><<<dim3(n_layers, chunks), 256, 0, s>>>(st, k0);
        if (rest > 0) {
            const unsigned t = (unsigned)((rest + 63) / 64);
            note_launches(1);
            update_kernel<TS><<<dim3(t, t, n_layers), 256, 0, s>>>(st, k0);
        }
    }
    return cudaGetLastError();
}

template <typename TS, int G>
cudaError_t apply_impl(int n_layers, int64_t D, const void* state, const float* q, int64_t n_q, int64_t ld_q,
                       void* qhat, int64_t ld_qhat, cudaStream_t s) {
    St<TS> st = state_of<TS>(const_cast<void*>(state), D);
    const size_t smem = (size_t)G * D * sizeof(TS);
    cudaError_t e = cudaFuncSetAttribute(apply_kernel<TS, G>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         (int)smem);
    if (e != cudaSuccess) return e;
    note_launches(1);
    apply_kernel<TS, G><<<dim3((unsigned)((n_q + G - 1) / G), n_layers), 256, smem, s>>>(st, q, n_q, ld_q,
                                                                                     (TS*)qhat, ld_qhat);
    return cudaGetLastError();
}

// ---------------------------------------------------------------- blocked path (fp32)
constexpr int kBB = 128;                // panel width
constexpr int64_t kBlockedMinD = 2048;  // smaller layers keep the one-launch cluster path
constexpr int kTrsmWarps = 8;
constexpr size_t kDiagSmem = sizeof(float) * (size_t)kBB * (kBB + 1);
constexpr size_t kTrsmSmem =
    sizeof(float) * ((size_t)kBB * (kBB + 1) + (size_t)(kBB / kNB) * kNB * (kNB + 1) + (size_t)kTrsmWarps * kBB);

// Factor the 128 x 128 diagonal block at lo of every layer (grid = layer) in
// shared memory by the left-looking (Cholesky-Crout) order, one column per
// step: L_ij = (A_ij - sum_{m<j} L_im L_jm) / L_jj for every row i >= j at
// once, two threads per row (each half of the dot product, four independent
// partial sums). The serial chain is one short dot product, one rsqrt and two
// barriers per column. L returns to M's lower triangle; the inverses of the
// four 32 x 32 diagonal blocks go to Dinv (one warp each); a non-positive
// pivot is recorded in the header and its column turns NaN.
__global__ void __launch_bounds__(256) diag_block_kernel(St<float> st, int64_t lo) {
    extern __shared__ __align__(16) float dsm[];
    float(*A)[kBB + 1] = reinterpret_cast<float(*)[kBB + 1]>(dsm);
    __shared__ float sinv[kBB];
    const int l = blockIdx.x;
    const int64_t D = st.D;
    float* M = st.M(l);
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    for (int e = tid; e < kBB * kBB; e += 256) {
        const int i = e / kBB, j = e % kBB;
        A[i][j] = (j <= i) ? M[(lo + i) * D + lo + j] : 0.f;
    }
    __syncthreads();
    const int i = tid >> 1, h = tid & 1;
#pragma unroll 1
    for (int j = 0; j < kBB; ++j) {
        float s = 0.f;
        if (i >= j) {
            float a0 = 0.f, a1 = 0.f, a2 = 0.f, a3 = 0.f;
            int m = h;
            for (; m + 6 < j; m += 8) {
                a0 = fmaf(A[i][m], A[j][m], a0);
                a1 = fmaf(A[i][m + 2], A[j][m + 2], a1);
                a2 = fmaf(A[i][m + 4], A[j][m + 4], a2);
                a3 = fmaf(A[i][m + 6], A[j][m + 6], a3);
            }
            for (; m < j; m += 2) a0 = fmaf(A[i][m], A[j][m], a0);
            s = (a0 + a1) + (a2 + a3);
        }
        s += __shfl_xor_sync(0xffffffffu, s, 1);
        s = (i >= j) ? A[i][j] - s : 0.f;
        if (i == j && h == 0) {
            const bool ok = s > 0.f;
            if (!ok) {
                double* hd = st.header(l);
                if (hd[kPcFailedPivot] == 0.0) hd[kPcFailedPivot] = (double)(lo + j + 1);
            }
            // L_jj = s * rsqrt(s), 1 / L_jj = rsqrt(s)
            const float inv = ok ? rsqrtf(s) : NAN;
            sinv[j] = inv;
            A[j][j] = s * inv;
        }
        __syncthreads();
        if (i > j && h == 0) A[i][j] = s * sinv[j];
        __syncthreads();
    }
    // inverses of the four diagonal blocks: warp w, lane c solves L X[:, c] = e_c
    if (warp < kBB / kNB) {
        const int b0 = warp * kNB, c = lane;
        float x[kNB];
#pragma unroll
        for (int r = 0; r < kNB; ++r) x[r] = (r == c) ? 1.f : 0.f;
#pragma unroll
        for (int jj = 0; jj < kNB; ++jj) {
            x[jj] = (jj < c) ? 0.f : x[jj] * sinv[b0 + jj];
#pragma unroll
            for (int r = jj + 1; r < kNB; ++r) x[r] -= A[b0 + r][b0 + jj] * x[jj];
        }
        float* Dg = st.Dinv(l) + ((lo + b0) / kNB) * (kNB * kNB);
#pragma unroll
        for (int r = 0; r < kNB; ++r) Dg[r * kNB + c] = x[r];
    }
    for (int e = tid; e < kBB * kBB; e += 256) {
        const int r = e / kBB, c = e % kBB;
        if (c <= r) M[(lo + r) * D + lo + c] = A[r][c];
    }
}

// Triangular solves of row vectors against the diagonal block B at lo of layer
// l (grid y): FWD x <- L_BB^{-1} x, else x <- L_BB^{-T} x, for n_rows rows of
// 128 values at column lo of X (row stride ldx, layer l's rows at byte offset
// l * layer_bytes from base). One warp per row; the block's L and its four
// diagonal inverses sit in shared memory. Used for the panel (rows of M below
// the block, FWD) and for the query rows of APPLY (both directions).
template <bool FWD>
__global__ void __launch_bounds__(256) trsm_block_kernel(St<float> st, int64_t lo, char* base, size_t layer_bytes,
                                                         int64_t ldx, int64_t n_rows) {
    extern __shared__ __align__(16) float tsm[];
    float(*Lb)[kBB + 1] = reinterpret_cast<float(*)[kBB + 1]>(tsm);
    float(*Di)[kNB][kNB + 1] = reinterpret_cast<float(*)[kNB][kNB + 1]>(tsm + kBB * (kBB + 1));
    float* Y = tsm + kBB * (kBB + 1) + (kBB / kNB) * kNB * (kNB + 1);
    const int l = blockIdx.y;
    const int64_t D = st.D;
    const float* M = st.M(l);
    const float* Dv = st.Dinv(l) + (lo / kNB) * (kNB * kNB);
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    for (int e = tid; e < kBB * kBB; e += 256) {
        const int i = e / kBB, j = e % kBB;
        Lb[i][j] = (j <= i) ? M[(lo + i) * D + lo + j] : 0.f;
    }
    for (int e = tid; e < (kBB / kNB) * kNB * kNB; e += 256) {
        const int b = e / (kNB * kNB), i = (e / kNB) % kNB, j = e % kNB;
        Di[b][i][j] = Dv[e];
    }
    __syncthreads();
    float* y = Y + warp * kBB;
    float* X = (float*)(base + (size_t)l * layer_bytes);
    for (int64_t r = (int64_t)blockIdx.x * kTrsmWarps + warp; r < n_rows; r += (int64_t)gridDim.x * kTrsmWarps) {
        float* x = X + r * ldx + lo;
#pragma unroll
        for (int c = lane; c < kBB; c += 32) y[c] = x[c];
        __syncwarp();
        if (FWD) {
#pragma unroll 1
            for (int b = 0; b < kBB / kNB; ++b) {
                const int c0 = b * kNB;
                float acc = y[c0 + lane];
                for (int m = 0; m < c0; ++m) acc -= Lb[c0 + lane][m] * y[m];
                float out = 0.f;
#pragma unroll
                for (int m = 0; m < kNB; ++m) {
                    const float rm = __shfl_sync(0xffffffffu, acc, m);
                    if (m <= lane) out += Di[b][lane][m] * rm;
                }
                __syncwarp();
                y[c0 + lane] = out;
                __syncwarp();
            }
        } else {
#pragma unroll 1
            for (int b = kBB / kNB - 1; b >= 0; --b) {
                const int c0 = b * kNB;
                float acc = y[c0 + lane];
                for (int m = c0 + kNB; m < kBB; ++m) acc -= Lb[m][c0 + lane] * y[m];
                float out = 0.f;
#pragma unroll
                for (int j = 0; j < kNB; ++j) {
                    const float rj = __shfl_sync(0xffffffffu, acc, j);
                    if (j >= lane) out += Di[b][j][lane] * rj;
                }
                __syncwarp();
                y[c0 + lane] = out;
                __syncwarp();
            }
        }
#pragma unroll
        for (int c = lane; c < kBB; c += 32) x[c] = y[c];
        __syncwarp();
    }
}

// Lower triangle of M <- M / n_total + lambda I for the blocked path: one row per
// loop step of a CTA, the row's columns across the threads (coalesced, no per-element
// index division). grid (row groups, layer).
__global__ void __launch_bounds__(256) scale_lower_kernel(St<float> st) {
    const int l = blockIdx.y;
    const int64_t D = st.D;
    const double* h = st.header(l);
    const float inv_n = (float)(1.0 / h[kPcNTotal]), lam = (float)h[kPcLambda];
    float* M = st.M(l);
    for (int64_t a = blockIdx.x; a < D; a += gridDim.x) {
        float* row = M + a * D;
        for (int64_t b = threadIdx.x; b <= a; b += 256) {
            float v = row[b] * inv_n;
            if (b == a) v += lam;
            row[b] = v;
        }
    }
}

// M[i][j] = M[j][i] for every 32 x 32 block strictly above the diagonal blocks
// (U = L^T, read by the backward solve's tensor-core products).
__global__ void __launch_bounds__(256) upper_from_lower_kernel(St<float> st, int n_layers) {
    __shared__ float t[kNB][kNB + 1];
    const int64_t D = st.D, nb = D / kNB, pairs = nb * (nb - 1) / 2;
    const int tx = threadIdx.x & 31, ty = threadIdx.x >> 5;
    for (int64_t w = blockIdx.x; w < pairs * n_layers; w += gridDim.x) {
        const int l = (int)(w / pairs);
        const int64_t p = w - (int64_t)l * pairs;
        int64_t bj = (int64_t)((1.0 + sqrt(1.0 + 8.0 * (double)p)) * 0.5);  // p = bj(bj-1)/2 + bi, bi < bj
        while (bj * (bj - 1) / 2 > p) --bj;
        while ((bj + 1) * bj / 2 <= p) ++bj;
        const int64_t bi = p - bj * (bj - 1) / 2;
        float* M = st.M(l);
        for (int r = ty; r < kNB; r += 8) t[r][tx] = M[(bj * kNB + r) * D + bi * kNB + tx];
        __syncthreads();
        for (int r = ty; r < kNB; r += 8) M[(bi * kNB + r) * D + bj * kNB + tx] = t[tx][r];
        __syncthreads();
    }
}

// Query rows of a layer whose factorisation failed become NaN.
__global__ void nan_failed_kernel(St<float> st, float* qhat, int64_t ld, int64_t n_q) {
    const int l = blockIdx.y;
    if (st.header(l)[kPcFailedPivot] == 0.0) return;
    const int64_t D = st.D;
    for (int64_t e = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; e < n_q * D; e += (int64_t)gridDim.x * blockDim.x)
        qhat[(e / D) * ld + (int64_t)l * D + e % D] = NAN;
}

bool blocked_pc(int64_t D, tda_dtype sdt) {
    return sdt == TDA_F32 && D % kBB == 0 && D >= kBlockedMinD && D < (1LL << 31) / kBB && gemm_tc_available();
}

cudaError_t blocked_attrs() {
    static cudaError_t e = [] {
        cudaError_t r = cudaFuncSetAttribute(diag_block_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                             (int)kDiagSmem);
        if (r == cudaSuccess)
            r = cudaFuncSetAttribute(trsm_block_kernel<true>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                     (int)kTrsmSmem);
        if (r == cudaSuccess)
            r = cudaFuncSetAttribute(trsm_block_kernel<false>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                     (int)kTrsmSmem);
        return r;
    }();
    return e;
}

unsigned trsm_grid(int64_t n_rows, int n_layers) {
    int64_t g = (n_rows + kTrsmWarps - 1) / kTrsmWarps;
    const int64_t cap = n_layers >= 304 ? 1 : 304 / n_layers;  // about two CTAs per SM over all layers
    if (g > cap) g = cap;
    return (unsigned)(g < 1 ? 1 : g);
}

cudaError_t factor_blocked(int n_layers, int64_t D, void* state, int64_t n_total, double la, double lr,
                           cudaStream_t s) {
    cudaError_t e = blocked_attrs();
    if (e != cudaSuccess) return e;
    unsigned int* err = device_error_word();
    if (!err) return cudaErrorUnknown;
    St<float> st = state_of<float>(state, D);
    note_launches(2);
    prepare_kernel<float><<<n_layers, 256, 0, s>>>(st, n_total, la, lr);
    const unsigned rows_per = (unsigned)((D < 1024 ? D : 1024) * (n_layers < 8 ? 8 / n_layers : 1));
    scale_lower_kernel<<<dim3(rows_per < (unsigned)D ? rows_per : (unsigned)D, n_layers), 256, 0, s>>>(st);
    // outer panels of 256 columns, each two 128-column sub-panels: the second sub-panel's
    // columns take the first one's update alone (a 128-wide product), and the trailing
    // matrix takes both at once (rank-256 update: twice the work per tile pass over M)
    float* M0 = (float*)((char*)state + 64);  // layer l's M is st.bytes further on
    const int64_t cz = (int64_t)(st.bytes / 4);
    for (int64_t lo = 0; lo < D; lo += 2 * kBB) {
        const int64_t mid = lo + kBB;
        note_launches(1);
        diag_block_kernel<<<n_layers, 256, kDiagSmem, s>>>(st, lo);
        if (mid == D) break;
        note_launches(1);
        trsm_block_kernel<true><<<dim3(trsm_grid(D - mid, n_layers), n_layers), 256, kTrsmSmem, s>>>(
            st, lo, (char*)M0 + (size_t)mid * D * 4, st.bytes, D, D - mid);
        // rows [mid, D) of columns [mid, mid + 128) -= L[rows, lo:mid] L[mid:mid+128, lo:mid]^T
        e = launch_gemm_nt_tc_batched(M0 + mid * D + lo, kBB, D, st.bytes, M0 + mid * D + lo, D - mid, D, st.bytes,
                                      kBB, M0 + mid * D + mid, D, cz, n_layers, -1.f, 1.f, false, err, s);
        if (e != cudaSuccess) return e;
        note_launches(1);
        diag_block_kernel<<<n_layers, 256, kDiagSmem, s>>>(st, mid);
        const int64_t hi = mid + kBB, rest = D - hi;
        if (rest == 0) break;
        note_launches(1);
        trsm_block_kernel<true><<<dim3(trsm_grid(rest, n_layers), n_layers), 256, kTrsmSmem, s>>>(
            st, mid, (char*)M0 + (size_t)hi * D * 4, st.bytes, D, rest);
        // trailing lower triangle of all layers in one launch: M -= P P^T, P = L[hi:D, lo:hi]
        e = launch_gemm_nt_tc_batched(M0 + hi * D + lo, rest, D, st.bytes, M0 + hi * D + lo, rest, D, st.bytes,
                                      2 * kBB, M0 + hi * D + hi, D, cz, n_layers, -1.f, 1.f, true, err, s);
        if (e != cudaSuccess) return e;
    }
    const int64_t nb = D / kNB;
    int64_t g = nb * (nb - 1) / 2 * n_layers;
    if (g > 152 * 8) g = 152 * 8;
    note_launches(1);
    upper_from_lower_kernel<<<(unsigned)g, 256, 0, s>>>(st, n_layers);
    return cudaGetLastError();
}

bool apply_blocked_ok(int64_t D, tda_dtype sdt, const void* qhat, int64_t ld_qhat, int64_t n_q) {
    return blocked_pc(D, sdt) && ((uintptr_t)qhat & 15) == 0 && (ld_qhat & 3) == 0 && n_q < (1LL << 24);
}

cudaError_t apply_blocked(int n_layers, int64_t D, const void* state, const float* q, int64_t n_q, int64_t ld_q,
                          float* qhat, int64_t ld_qhat, cudaStream_t s) {
    cudaError_t e = blocked_attrs();
    if (e != cudaSuccess) return e;
    unsigned int* err = device_error_word();
    if (!err) return cudaErrorUnknown;
    St<float> st = state_of<float>(const_cast<void*>(state), D);
    if (q != qhat || ld_q != ld_qhat) {
        e = cudaMemcpy2DAsync(qhat, (size_t)ld_qhat * 4, q, (size_t)ld_q * 4, (size_t)n_layers * D * 4, (size_t)n_q,
                              cudaMemcpyDeviceToDevice, s);
        if (e != cudaSuccess) return e;
    }
    const unsigned gx = trsm_grid(n_q, n_layers);
    const size_t lb = (size_t)D * 4;  // layer l's columns start l * D floats into each row
    const float* M0 = (const float*)((const char*)state + 64);  // layer l's M is st.bytes further on
    for (int64_t lo = 0; lo < D; lo += kBB) {
        note_launches(1);
        trsm_block_kernel<true><<<dim3(gx, n_layers), 256, kTrsmSmem, s>>>(st, lo, (char*)qhat, lb, ld_qhat, n_q);
        const int64_t hi = lo + kBB;
        if (hi == D) break;
        e = launch_gemm_nt_tc_batched(M0 + hi * D + lo, D - hi, D, st.bytes, qhat + lo, n_q, ld_qhat, lb, kBB,
                                      qhat + hi, ld_qhat, D, n_layers, -1.f, 1.f, false, err, s);
        if (e != cudaSuccess) return e;
    }
    for (int64_t lo = D - kBB; lo >= 0; lo -= kBB) {
        note_launches(1);
        trsm_block_kernel<false><<<dim3(gx, n_layers), 256, kTrsmSmem, s>>>(st, lo, (char*)qhat, lb, ld_qhat, n_q);
        if (lo == 0) break;
        // rows [0, lo) of U = L^T, columns [lo, lo + 128): U[i][j] = L[j][i]
        e = launch_gemm_nt_tc_batched(M0 + lo, lo, D, st.bytes, qhat + lo, n_q, ld_qhat, lb, kBB, qhat, ld_qhat, D,
                                      n_layers, -1.f, 1.f, false, err, s);
        if (e != cudaSuccess) return e;
    }
    note_launches(1);
    nan_failed_kernel<<<dim3(64, n_layers), 256, 0, s>>>(st, qhat, ld_qhat, n_q);
    return cudaGetLastError();
}

}  // namespace

int64_t precondition_apply_max_d(tda_dtype sdt) {
    // one query row of D elements must fit the shared-memory budget of APPLY
    return (int64_t)(160 * 1024) / (sdt == TDA_F64 ? 8 : 4);
}

cudaError_t launch_pc_fit(int n_layers, int64_t D, tda_dtype sdt, void* state, const float* phi, int64_t n,
                          int64_t ld, cudaStream_t s) {
    if (n == 0) return cudaSuccess;
    if (sdt == TDA_F32 && fit_tc_supported(n_layers, D, phi, n, ld)) {
        unsigned int* err = device_error_word();
        if (err)
            return launch_fit_tc(n_layers, D, state, tda_precondition_state_bytes(D, TDA_F32), phi, n, ld, err, s);
    }
    note_launches(1);
    if (sdt == TDA_F64) {
        const unsigned t = (unsigned)((D + 63) / 64);
        fit_f64_kernel<<<dim3(t, t, n_layers), 256, 0, s>>>(state_of<double>(state, D), phi, n, ld);
    } else {
        const unsigned t = (unsigned)((D + kFT - 1) / kFT);
        fit_f32_kernel<<<dim3(t, t, n_layers), 256, 0, s>>>(state_of<float>(state, D), phi, n, ld);
    }
    return cudaGetLastError();
}

cudaError_t launch_pc_factor(int n_layers, int64_t D, tda_dtype sdt, void* state, int64_t n_total,
                             double lambda_abs, double lambda_rel, cudaStream_t s) {
    if (blocked_pc(D, sdt)) return factor_blocked(n_layers, D, state, n_total, lambda_abs, lambda_rel, s);
    if (sdt == TDA_F64) return factor_impl<double>(n_layers, D, state, n_total, lambda_abs, lambda_rel, s);
    return factor_impl<float>(n_layers, D, state, n_total, lambda_abs, lambda_rel, s);
}

cudaError_t launch_pc_factor_apply(int n_layers, int64_t D, tda_dtype sdt, void* state, int64_t n_total,
                                   double lambda_abs, double lambda_rel, const float* q, int64_t n_q, int64_t ld_q,
                                   void* qhat, int64_t ld_qhat, cudaStream_t s) {
    // fp32 state, whole 32-column blocks, up to 256 queries: factorisation and both
    // substitutions in one cluster launch per call (below the blocked path's sizes);
    // otherwise FACTOR, then APPLY
    if (sdt == TDA_F32 && !blocked_pc(D, sdt) && D % kNB == 0 && D >= 2 * kNB && n_q >= 1 && n_q <= 256) {
        const QArgs qa{q, (float*)qhat, n_q, ld_q, ld_qhat};
        cudaError_t e = factor_cluster<16, true>(n_layers, D, state, n_total, lambda_abs, lambda_rel, qa, s);
        if (e == cudaErrorNotSupported)
            e = factor_cluster<8, true>(n_layers, D, state, n_total, lambda_abs, lambda_rel, qa, s);
        if (e != cudaErrorNotSupported) return e;
    }
    cudaError_t e = launch_pc_factor(n_layers, D, sdt, state, n_total, lambda_abs, lambda_rel, s);
    if (e != cudaSuccess) return e;
    return launch_pc_apply(n_layers, D, sdt, state, q, n_q, ld_q, qhat, ld_qhat, s);
}

cudaError_t launch_pc_apply(int n_layers, int64_t D, tda_dtype sdt, const void* state, const float* q,
                            int64_t n_q, int64_t ld_q, void* qhat, int64_t ld_qhat, cudaStream_t s) {
    if (n_q == 0) return cudaSuccess;
    // a blocked factorisation left L^T in M's upper triangle: tensor-core substitutions
    if (apply_blocked_ok(D, sdt, qhat, ld_qhat, n_q))
        return apply_blocked(n_layers, D, state, q, n_q, ld_q, (float*)qhat, ld_qhat, s);
    const size_t el = sdt == TDA_F64 ? 8 : 4;
    const size_t budget = 160 * 1024;
    if (sdt == TDA_F64) {
        if ((size_t)D * el * 8 <= budget)
            return apply_impl<double, 8>(n_layers, D, state, q, n_q, ld_q, qhat, ld_qhat, s);
        if ((size_t)D * el * 2 <= budget)
            return apply_impl<double, 2>(n_layers, D, state, q, n_q, ld_q, qhat, ld_qhat, s);
        return apply_impl<double, 1>(n_layers, D, state, q, n_q, ld_q, qhat, ld_qhat, s);
    }
    if ((size_t)D * el * 4 <= budget) return apply_impl<float, 4>(n_layers, D, state, q, n_q, ld_q, qhat, ld_qhat, s);
    if ((size_t)D * el * 2 <= budget) return apply_impl<float, 2>(n_layers, D, state, q, n_q, ld_q, qhat, ld_qhat, s);
    return apply_impl<float, 1>(n_layers, D, state, q, n_q, ld_q, qhat, ld_qhat, s);
}

}  // namespace tda
