// k_kfac.cu -- K-FAC and EK-FAC on projected factors (the paper applies both
// Kronecker-factored curvature methods to the projected pair (a~, g~)
// unchanged, App. A.2, and damps by a multiple of the mean eigenvalue,
// App. B.2):
//   factor covariances  C_a = (1/M) sum a~ a~^T, C_g = (1/M) sum g~ g~^T,
//   eigenbases          C = U diag(w) U^T (parallel cyclic Jacobi, fp64),
//   EK-FAC eigenvalues  Lam = (1/N) sum_i (U_g^T Phi_i U_a)^2,
//   preconditioning     Qhat = U_g [(U_g^T Q U_a) / (Lam + lambda)] U_a^T.
// Sums over examples go through per-CTA partials reduced in a fixed order, so
// results do not depend on scheduling.
#include "tda_internal.cuh"

namespace tda {

// fp64 state of one layer, offsets in doubles
struct KfLayout {
    int64_t ka, kg, Sa, Sg, Ua, wa, Ug, wg, Le, total;
    __host__ __device__ explicit KfLayout(int64_t k_in, int64_t k_out) : ka(k_in), kg(k_out) {
        Sa = 8;  // header: [0] M token positions, [1] N examples (EK-FAC), [2] Jacobi sweeps a, [3] sweeps g
        Sg = Sa + ka * ka;
        Ua = Sg + kg * kg;
        wa = Ua + ka * ka;
        Ug = wa + ka;
        wg = Ug + kg * kg;
        Le = wg + kg;
        total = Le + ka * kg;
    }
};

size_t kfac_state_bytes(int64_t k_in, int64_t k_out) {
    const KfLayout l(k_in, k_out);
    return ((size_t)l.total * 8 + 255) & ~(size_t)255;
}

namespace {

constexpr int kKfThreads = 256;

// part[b][i*k+j] = sum over the rows of block b of Y[r][i] * Y[r][j] (fp32)
__global__ void __launch_bounds__(kKfThreads)
cov_partial_kernel(const float* __restrict__ Y, int64_t rows, int k, int64_t rows_per_block, float* __restrict__ part) {
    extern __shared__ float ys[];  // [64][k]
    const int64_t r0 = (int64_t)blockIdx.x * rows_per_block;
    int64_t r1 = r0 + rows_per_block;
    if (r1 > rows) r1 = rows;
    const int kk = k * k;
    constexpr int kMaxPer = 64;  // k <= 128: k*k / 256 <= 64 entries per thread
    float acc[kMaxPer];
#pragma unroll
    for (int m = 0; m < kMaxPer; ++m) acc[m] = 0.f;
    for (int64_t b0 = r0; b0 < r1; b0 += 64) {
        const int nr = (int)((r1 - b0) < 64 ? (r1 - b0) : 64);
        __syncthreads();
        for (int x = threadIdx.x; x < nr * k; x += blockDim.x) ys[x] = Y[b0 * k + x];
        __syncthreads();
#pragma unroll
        for (int m = 0; m < kMaxPer; ++m) {
            const int e = threadIdx.x + m * kKfThreads;
            if (e < kk) {
                const int i = e / k, j = e - (e / k) * k;
                float a = acc[m];
                for (int r = 0; r < nr; ++r) a = fmaf(ys[r * k + i], ys[r * k + j], a);
                acc[m] = a;
            }
        }
    }
    float* out = part + (int64_t)blockIdx.x * kk;
#pragma unroll
    for (int m = 0; m < kMaxPer; ++m) {
        const int e = threadIdx.x + m * kKfThreads;
        if (e < kk) out[e] = acc[m];
    }
}

// S[e] += scale * sum_b part[b * stride + e] in block order (fp64); header[slot] += add
__global__ void sum_partials_kernel(const float* __restrict__ part, int nblk, int64_t stride, int64_t n,
                                    double* __restrict__ S, double scale, double* __restrict__ header, int slot,
                                    double add) {
    for (int64_t e = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; e < n; e += (int64_t)gridDim.x * blockDim.x) {
        double v = 0.0;
        for (int b = 0; b < nblk; ++b) v += (double)part[(int64_t)b * stride + e];
        S[e] += scale * v;
    }
    if (header && blockIdx.x == 0 && threadIdx.x == 0) header[slot] += add;
}

__device__ __forceinline__ float j_sqrt(float x) { return sqrtf(x); }
__device__ __forceinline__ double j_sqrt(double x) { return sqrt(x); }
__device__ __forceinline__ float j_abs(float x) { return fabsf(x); }
__device__ __forceinline__ double j_abs(double x) { return fabs(x); }

// Parallel cyclic Jacobi (round-robin pair ordering) by one CTA on the
// symmetric n x n matrix A in shared memory (row stride lda), accumulating
// V <- V J (row stride ldv). Each round rotates floor(m/2) disjoint pairs at
// once: angles from the round's starting matrix, then all row updates, then
// all column updates, which is J^T A J for the product J of the round's
// rotations. Stops when the off-diagonal squared norm is <= tol * fro (fro =
// squared norm of A at entry); returns the sweep count, or -1 after
// max_sweeps. Shared matrices use an odd row stride (n + 1) so that the column
// updates, whose threads walk down a column, hit distinct banks.
template <typename T>
__device__ int jacobi_sweeps(T* A, int lda, T* V, int ldv, int n, T* cs, T* sn, int* P, int* Q, double* red, int* done,
                             double tol, int max_sweeps) {
    const int m = (n + 1) & ~1;  // even number of players; index n is a dummy when n is odd
    double f = 0.0;
    for (int e = threadIdx.x; e < n * n; e += blockDim.x) {
        const double a = (double)A[(e / n) * lda + e % n];
        f += a * a;
    }
    red[threadIdx.x] = f;
    __syncthreads();
    for (int h = blockDim.x / 2; h > 0; h >>= 1) {
        if (threadIdx.x < h) red[threadIdx.x] += red[threadIdx.x + h];
        __syncthreads();
    }
    const double fro = red[0];
    __syncthreads();
    int sweep = 0;
    for (; sweep < max_sweeps; ++sweep) {
        double off = 0.0;
        for (int e = threadIdx.x; e < n * n; e += blockDim.x)
            if (e / n != e % n) {
                const double a = (double)A[(e / n) * lda + e % n];
                off += a * a;
            }
        red[threadIdx.x] = off;
        __syncthreads();
        for (int h = blockDim.x / 2; h > 0; h >>= 1) {
            if (threadIdx.x < h) red[threadIdx.x] += red[threadIdx.x + h];
            __syncthreads();
        }
        if (threadIdx.x == 0) *done = (red[0] <= tol * fro) ? 1 : 0;
        __syncthreads();
        if (*done) return sweep;
        for (int r = 0; r < m - 1; ++r) {
            for (int i = threadIdx.x; i < m / 2; i += blockDim.x) {
                int p = i == 0 ? r : (r + i) % (m - 1);
                int q = i == 0 ? m - 1 : (r - i + m - 1) % (m - 1);
                if (p > q) {
                    const int t = p;
                    p = q;
                    q = t;
                }
                T c = 1, sv = 0;
                if (q < n) {
                    const T apq = A[p * lda + q];
                    if (apq != T(0)) {
                        const T tau = (A[q * lda + q] - A[p * lda + p]) / (T(2) * apq);
                        const T t = (tau >= T(0) ? T(1) : T(-1)) / (j_abs(tau) + j_sqrt(T(1) + tau * tau));
                        c = T(1) / j_sqrt(T(1) + t * t);
                        sv = t * c;
                    }
                }
                cs[i] = c;
                sn[i] = sv;
                P[i] = p;
                Q[i] = q < n ? q : -1;
            }
            __syncthreads();
            const int half = m / 2;
            for (int x = threadIdx.x; x < half * n; x += blockDim.x) {  // rows p, q: A <- J^T A
                const int i = x / n, k = x - (x / n) * n;
                if (Q[i] < 0 || sn[i] == T(0)) continue;
                const int p = P[i], q = Q[i];
                const T c = cs[i], sv = sn[i], apk = A[p * lda + k], aqk = A[q * lda + k];
                A[p * lda + k] = c * apk - sv * aqk;
                A[q * lda + k] = sv * apk + c * aqk;
            }
            __syncthreads();
            for (int x = threadIdx.x; x < half * n; x += blockDim.x) {  // columns p, q: A <- A J, V <- V J
                const int i = x / n, k = x - (x / n) * n;
                if (Q[i] < 0 || sn[i] == T(0)) continue;
                const int p = P[i], q = Q[i];
                const T c = cs[i], sv = sn[i];
                const T akp = A[k * lda + p], akq = A[k * lda + q];
                A[k * lda + p] = c * akp - sv * akq;
                A[k * lda + q] = sv * akp + c * akq;
                const T vkp = V[k * ldv + p], vkq = V[k * ldv + q];
                V[k * ldv + p] = c * vkp - sv * vkq;
                V[k * ldv + q] = sv * vkp + c * vkq;
            }
            __syncthreads();
        }
    }
    return -1;
}

// out = X^T Y (tx) or X Y, n x n fp64 in shared memory, row stride ld (one CTA)
__device__ void gemm_nn(double* out, const double* X, const double* Y, int n, int ld, bool tx) {
    for (int e = threadIdx.x; e < n * n; e += blockDim.x) {
        const int i = e / n, j = e - (e / n) * n;
        double acc = 0.0;
        for (int k = 0; k < n; ++k) acc += (tx ? X[k * ld + i] : X[i * ld + k]) * Y[k * ld + j];
        out[i * ld + j] = acc;
    }
    __syncthreads();
}

// Eigenbases of C = S / M for the a side (blockIdx.x 0) and the g side (1) of
// layer blockIdx.y, C = U diag(w) U^T.
//   n <= 64 (MIXED): the sweeps run in fp32 (the fp64 pipe is a small fraction
//   of the fp32 one here) until the off-diagonal part is near fp32 rounding;
//   then, in fp64, two Newton-Schulz steps V <- V (3I - V^T V) / 2 make the
//   fp32 eigenvectors orthonormal to fp64 precision, A = V^T C V is formed
//   afresh, and fp64 sweeps finish (typically two). The header gets the fp64
//   sweep count.
//   n > 64: fp64 sweeps from the start, V in the state's U.
template <bool MIXED>
__global__ void __launch_bounds__(kKfThreads)
jacobi_kernel(double* __restrict__ st0, int64_t stride, int64_t ka, int64_t kg) {
    extern __shared__ double smd[];
    double* st = st0 + (int64_t)blockIdx.y * stride;
    const KfLayout l(ka, kg);
    const bool side_g = blockIdx.x == 1;
    const int n = (int)(side_g ? kg : ka);
    const double* S = st + (side_g ? l.Sg : l.Sa);
    double* U = st + (side_g ? l.Ug : l.Ua);
    double* w = st + (side_g ? l.wg : l.wa);
    const int nmax = (int)(ka > kg ? ka : kg), mh = (nmax + 2) / 2, ld = n + 1, sq = nmax * (nmax + 1);
    __shared__ double red[kKfThreads];
    __shared__ int done;
    const double Mtok = st[0];
    const double inv = Mtok > 0 ? 1.0 / Mtok : 0.0;
    double* A = smd;  // [n][ld]
    int sweeps;
    if constexpr (MIXED) {
        double* V = A + sq;
        double* Tm = V + sq;  // fp64 scratch
        double* cs = Tm + sq;
        double* sn = cs + mh;
        float* A32 = (float*)(sn + mh);
        float* V32 = A32 + sq;
        float* cs32 = V32 + sq;
        float* sn32 = cs32 + mh;
        int* P = (int*)(sn32 + mh);
        int* Q = P + mh;
        for (int e = threadIdx.x; e < n * n; e += blockDim.x) {
            const int i = e / n, j = e % n;
            A32[i * ld + j] = (float)(S[e] * inv);
            V32[i * ld + j] = (i == j) ? 1.f : 0.f;
        }
        __syncthreads();
        // fp32: the off-diagonal part down to about 1e-6 of ||C|| (near fp32 rounding; at most
        // 20 sweeps, since fp32 cannot go much further)
        jacobi_sweeps<float>(A32, ld, V32, ld, n, cs32, sn32, P, Q, red, &done, 1e-12, 20);
        for (int e = threadIdx.x; e < n * n; e += blockDim.x) {
            const int i = e / n, j = e % n;
            V[i * ld + j] = (double)V32[i * ld + j];
        }
        __syncthreads();
        for (int it = 0; it < 2; ++it) {  // Newton-Schulz: V <- V (3I - V^T V) / 2
            gemm_nn(Tm, V, V, n, ld, true);
            for (int e = threadIdx.x; e < n * n; e += blockDim.x) {
                const int i = e / n, j = e % n;
                Tm[i * ld + j] = ((i == j) ? 1.5 : 0.0) - 0.5 * Tm[i * ld + j];
            }
            __syncthreads();
            gemm_nn(A, V, Tm, n, ld, false);
            for (int e = threadIdx.x; e < n * n; e += blockDim.x) V[(e / n) * ld + e % n] = A[(e / n) * ld + e % n];
            __syncthreads();
        }
        for (int e = threadIdx.x; e < n * n; e += blockDim.x) A[(e / n) * ld + e % n] = S[e] * inv;  // C
        __syncthreads();
        gemm_nn(Tm, A, V, n, ld, false);  // C V
        gemm_nn(A, V, Tm, n, ld, true);   // V^T C V
        sweeps = jacobi_sweeps<double>(A, ld, V, ld, n, cs, sn, P, Q, red, &done, 1e-28, 60);
        for (int e = threadIdx.x; e < n * n; e += blockDim.x) U[e] = V[(e / n) * ld + e % n];
    } else {
        const bool v_shared = nmax <= 64;
        double* V = v_shared ? A + sq : U;
        const int ldv = v_shared ? ld : n;
        double* cs = A + (v_shared ? 2 : 1) * sq;
        double* sn = cs + mh;
        int* P = (int*)(sn + mh);
        int* Q = P + mh;
        for (int e = threadIdx.x; e < n * n; e += blockDim.x) {
            const int i = e / n, j = e % n;
            A[i * ld + j] = S[e] * inv;
            V[i * ldv + j] = (i == j) ? 1.0 : 0.0;
        }
        __syncthreads();
        sweeps = jacobi_sweeps<double>(A, ld, V, ldv, n, cs, sn, P, Q, red, &done, 1e-28, 60);
        if (v_shared)
            for (int e = threadIdx.x; e < n * n; e += blockDim.x) U[e] = V[(e / n) * ld + e % n];
    }
    for (int i = threadIdx.x; i < n; i += blockDim.x) w[i] = A[i * ld + i];
    if (threadIdx.x == 0) st[2 + (side_g ? 1 : 0)] = (double)sweeps;
    if (blockIdx.x == 0) {  // a new eigenbasis invalidates the EK-FAC sums
        for (int64_t e = threadIdx.x; e < ka * kg; e += blockDim.x) st[l.Le + e] = 0.0;
        if (threadIdx.x == 0) st[1] = 0.0;
    }
}

// Eigenbases of one layer as fp32 in shared memory (SU) or read from the fp64
// state (large k).
template <bool SU>
struct Bases {
    const float* ua;
    const float* ug;
    const double* uad;
    const double* ugd;
    __device__ __forceinline__ float a(int64_t i) const { return SU ? ua[i] : (float)uad[i]; }
    __device__ __forceinline__ float g(int64_t i) const { return SU ? ug[i] : (float)ugd[i]; }
};

// part[layer][b][r*ka+c] = sum over the examples of block b of ((U_g^T Phi_i U_a)[r][c])^2
template <bool SU>
__global__ void __launch_bounds__(kKfThreads)
ekfac_partial_kernel(const float* __restrict__ phi, int64_t n, int64_t ld, const double* __restrict__ st0,
                     int64_t stride, int64_t ka, int64_t kg, float* __restrict__ part) {
    extern __shared__ float sm[];  // [U_a, U_g if SU] Phi_i [kg][ka], Y [kg][ka]
    const int layer = blockIdx.y;
    const double* st = st0 + (int64_t)layer * stride;
    const KfLayout l(ka, kg);
    const int64_t D = ka * kg;
    float* F = sm + (SU ? ka * ka + kg * kg : 0);
    float* Y = F + D;
    Bases<SU> U{sm, sm + ka * ka, st + l.Ua, st + l.Ug};
    if (SU) {
        for (int64_t e = threadIdx.x; e < ka * ka; e += blockDim.x) sm[e] = (float)st[l.Ua + e];
        for (int64_t e = threadIdx.x; e < kg * kg; e += blockDim.x) sm[ka * ka + e] = (float)st[l.Ug + e];
    }
    const float* ph = phi + (int64_t)layer * D;
    constexpr int kMaxPer = 64;
    float acc[kMaxPer];
#pragma unroll
    for (int m = 0; m < kMaxPer; ++m) acc[m] = 0.f;
    for (int64_t i = blockIdx.x; i < n; i += gridDim.x) {
        __syncthreads();
        for (int64_t e = threadIdx.x; e < D; e += blockDim.x) F[e] = ph[i * ld + e];
        __syncthreads();
        for (int64_t e = threadIdx.x; e < D; e += blockDim.x) {  // Y = Phi U_a
            const int64_t r = e / ka, c = e - (e / ka) * ka;
            float sacc = 0.f;
            for (int64_t j = 0; j < ka; ++j) sacc = fmaf(F[r * ka + j], U.a(j * ka + c), sacc);
            Y[e] = sacc;
        }
        __syncthreads();
#pragma unroll
        for (int m = 0; m < kMaxPer; ++m) {  // X = U_g^T Y, accumulate X^2
            const int64_t e = threadIdx.x + (int64_t)m * kKfThreads;
            if (e < D) {
                const int64_t r = e / ka, c = e - (e / ka) * ka;
                float sacc = 0.f;
                for (int64_t j = 0; j < kg; ++j) sacc = fmaf(U.g(j * kg + r), Y[j * ka + c], sacc);
                acc[m] = fmaf(sacc, sacc, acc[m]);
            }
        }
    }
    float* out = part + ((int64_t)layer * gridDim.x + blockIdx.x) * D;
#pragma unroll
    for (int m = 0; m < kMaxPer; ++m) {
        const int64_t e = threadIdx.x + (int64_t)m * kKfThreads;
        if (e < D) out[e] = acc[m];
    }
}

// Square k = 16, 32, 64: thread (column c, row group g) keeps U_a[:, c] and,
// per example, column c of Y = Phi U_a in registers; Phi and U_g^T rows are
// read from shared memory as warp broadcasts, so each multiply-add costs a
// quarter of a (vector) shared load.
template <int K>
__global__ void __launch_bounds__(256)
ekfac_reg_kernel(const float* __restrict__ phi, int64_t n, int64_t ld, const double* __restrict__ st0, int64_t stride,
                 float* __restrict__ part) {
    constexpr int RG = 256 / K;  // row groups
    constexpr int RPT = K / RG;  // rows per thread
    __shared__ __align__(16) float F[K * K];    // Phi_i [r][j]
    __shared__ __align__(16) float Y[K * K];    // Phi_i U_a [r][c]
    __shared__ __align__(16) float UgT[K * K];  // U_g^T [r][j]
    const int layer = blockIdx.y;
    const double* st = st0 + (int64_t)layer * stride;
    const KfLayout l(K, K);
    const int c = threadIdx.x % K, g = threadIdx.x / K;
    float ua[K];
#pragma unroll
    for (int j = 0; j < K; ++j) ua[j] = (float)st[l.Ua + j * K + c];
    for (int e = threadIdx.x; e < K * K; e += 256) UgT[e] = (float)st[l.Ug + (e % K) * K + e / K];
    float acc[RPT];
#pragma unroll
    for (int m = 0; m < RPT; ++m) acc[m] = 0.f;
    const float* ph = phi + (int64_t)layer * K * K;
    for (int64_t i = blockIdx.x; i < n; i += gridDim.x) {
        __syncthreads();
        for (int e = threadIdx.x; e < K * K / 4; e += 256)
            reinterpret_cast<float4*>(F)[e] = reinterpret_cast<const float4*>(ph + i * ld)[e];
        __syncthreads();
#pragma unroll
        for (int m = 0; m < RPT; ++m) {  // Y[r][c] = sum_j Phi[r][j] U_a[j][c]
            const int r = g + RG * m;
            float sacc = 0.f;
#pragma unroll
            for (int j = 0; j < K; j += 4) {
                const float4 f = *reinterpret_cast<const float4*>(F + r * K + j);
                sacc = fmaf(f.x, ua[j], sacc);
                sacc = fmaf(f.y, ua[j + 1], sacc);
                sacc = fmaf(f.z, ua[j + 2], sacc);
                sacc = fmaf(f.w, ua[j + 3], sacc);
            }
            Y[r * K + c] = sacc;
        }
        __syncthreads();
        float yc[K];
#pragma unroll
        for (int j = 0; j < K; ++j) yc[j] = Y[j * K + c];
#pragma unroll
        for (int m = 0; m < RPT; ++m) {  // X[r][c] = sum_j U_g[j][r] Y[j][c]; accumulate X^2
            const int r = g + RG * m;
            float sacc = 0.f;
#pragma unroll
            for (int j = 0; j < K; j += 4) {
                const float4 u = *reinterpret_cast<const float4*>(UgT + r * K + j);
                sacc = fmaf(u.x, yc[j], sacc);
                sacc = fmaf(u.y, yc[j + 1], sacc);
                sacc = fmaf(u.z, yc[j + 2], sacc);
                sacc = fmaf(u.w, yc[j + 3], sacc);
            }
            acc[m] = fmaf(sacc, sacc, acc[m]);
        }
    }
    float* out = part + ((int64_t)layer * gridDim.x + blockIdx.x) * K * K;
#pragma unroll
    for (int m = 0; m < RPT; ++m) out[(g + RG * m) * K + c] = acc[m];
}

// Le of every layer += its block partials (fixed order); N += n
__global__ void ekfac_reduce_kernel(const float* __restrict__ part, int nblk, double* __restrict__ st0, int64_t stride,
                                    int64_t ka, int64_t kg, double n) {
    const int layer = blockIdx.y;
    double* st = st0 + (int64_t)layer * stride;
    const KfLayout l(ka, kg);
    const int64_t D = ka * kg;
    const float* pl = part + (int64_t)layer * nblk * D;
    for (int64_t e = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; e < D; e += (int64_t)gridDim.x * blockDim.x) {
        double v = 0.0;
        for (int b = 0; b < nblk; ++b) v += (double)pl[(int64_t)b * D + e];
        st[l.Le + e] += v;
    }
    if (blockIdx.x == 0 && threadIdx.x == 0) st[1] += n;
}

// One CTA per (query row, layer): Qhat = U_g [(U_g^T Q U_a) / (Lam + lambda)] U_a^T
template <bool SU>
__global__ void __launch_bounds__(kKfThreads)
kfac_apply_kernel(int kind, const double* __restrict__ st0, int64_t stride, int64_t ka, int64_t kg,
                  double lambda_abs, double lambda_rel, const float* __restrict__ q, int64_t ld_q,
                  float* __restrict__ qhat, int64_t ld_qhat) {
    extern __shared__ float sm[];  // [U_a, U_g if SU] X [kg][ka], Y [kg][ka]
    const int layer = blockIdx.y;
    const double* st = st0 + (int64_t)layer * stride;
    const KfLayout l(ka, kg);
    const int64_t D = ka * kg;
    float* X = sm + (SU ? ka * ka + kg * kg : 0);
    float* Y = X + D;
    Bases<SU> U{sm, sm + ka * ka, st + l.Ua, st + l.Ug};
    if (SU) {
        for (int64_t e = threadIdx.x; e < ka * ka; e += blockDim.x) sm[e] = (float)st[l.Ua + e];
        for (int64_t e = threadIdx.x; e < kg * kg; e += blockDim.x) sm[ka * ka + e] = (float)st[l.Ug + e];
    }
    __shared__ double red[kKfThreads];
    const double nex = st[1];
    auto lam_of = [&](int64_t e) -> double {
        const int64_t r = e / ka, c = e - (e / ka) * ka;
        if (kind == 0) return st[l.wg + r] * st[l.wa + c];
        return nex > 0 ? st[l.Le + e] / nex : 0.0;
    };
    double sacc = 0.0;
    for (int64_t e = threadIdx.x; e < D; e += blockDim.x) sacc += lam_of(e);
    red[threadIdx.x] = sacc;
    __syncthreads();
    for (int h = blockDim.x / 2; h > 0; h >>= 1) {
        if (threadIdx.x < h) red[threadIdx.x] += red[threadIdx.x + h];
        __syncthreads();
    }
    const double lambda = lambda_abs + lambda_rel * red[0] / (double)D;
    const float* qi = q + (int64_t)blockIdx.x * ld_q + (int64_t)layer * D;
    for (int64_t e = threadIdx.x; e < D; e += blockDim.x) X[e] = qi[e];
    __syncthreads();
    for (int64_t e = threadIdx.x; e < D; e += blockDim.x) {  // Y = Q U_a
        const int64_t r = e / ka, c = e - (e / ka) * ka;
        float a = 0.f;
        for (int64_t j = 0; j < ka; ++j) a = fmaf(X[r * ka + j], U.a(j * ka + c), a);
        Y[e] = a;
    }
    __syncthreads();
    for (int64_t e = threadIdx.x; e < D; e += blockDim.x) {  // X = (U_g^T Y) / (Lam + lambda)
        const int64_t r = e / ka, c = e - (e / ka) * ka;
        float a = 0.f;
        for (int64_t j = 0; j < kg; ++j) a = fmaf(U.g(j * kg + r), Y[j * ka + c], a);
        X[e] = (float)((double)a / (lam_of(e) + lambda));
    }
    __syncthreads();
    for (int64_t e = threadIdx.x; e < D; e += blockDim.x) {  // Y = X U_a^T
        const int64_t r = e / ka, c = e - (e / ka) * ka;
        float a = 0.f;
        for (int64_t j = 0; j < ka; ++j) a = fmaf(X[r * ka + j], U.a(c * ka + j), a);
        Y[e] = a;
    }
    __syncthreads();
    float* out = qhat + (int64_t)blockIdx.x * ld_qhat + (int64_t)layer * D;
    for (int64_t e = threadIdx.x; e < D; e += blockDim.x) {  // Qhat = U_g Y
        const int64_t r = e / ka, c = e - (e / ka) * ka;
        float a = 0.f;
        for (int64_t j = 0; j < kg; ++j) a = fmaf(U.g(r * kg + j), Y[j * ka + c], a);
        out[e] = a;
    }
}

}  // namespace

int kfac_partial_blocks(int64_t rows) {
    int64_t b = (rows + 255) / 256;
    if (b > 304) b = 304;
    return b < 1 ? 1 : (int)b;
}

// S += scale * Y^T Y for rows x k fp32 rows Y (deterministic), header M += add_m.
cudaError_t launch_kfac_cov(const float* Y, int64_t rows, int k, double* S, double scale, double* header,
                            double add_m, float* part, cudaStream_t s) {
    if (rows == 0) {
        if (header && add_m != 0) {
            note_launches(1);
            sum_partials_kernel<<<1, 32, 0, s>>>(part, 0, 0, 0, S, scale, header, 0, add_m);
        }
        return cudaGetLastError();
    }
    const int nb = kfac_partial_blocks(rows);
    int64_t per = (rows + nb - 1) / nb;
    per = (per + 63) / 64 * 64;
    const int nblk = (int)((rows + per - 1) / per);
    note_launches(2);
    cov_partial_kernel<<<nblk, kKfThreads, (size_t)64 * k * 4, s>>>(Y, rows, k, per, part);
    sum_partials_kernel<<<(unsigned)((k * k + 255) / 256), 256, 0, s>>>(part, nblk, (int64_t)k * k, (int64_t)k * k,
                                                                       S, scale, header, 0, add_m);
    return cudaGetLastError();
}

// Sums of per-CTA partials written by another kernel (the fused projection).
cudaError_t launch_kfac_sum_partials(const float* part, int nblk, int64_t stride, int64_t n, double* S, double scale,
                                     double* header, int slot, double add, cudaStream_t s) {
    note_launches(1);
    int64_t blocks = (n + 255) / 256;
    if (blocks < 1) blocks = 1;
    sum_partials_kernel<<<(unsigned)blocks, 256, 0, s>>>(part, nblk, stride, n, S, scale, header, slot, add);
    return cudaGetLastError();
}

cudaError_t launch_kfac_eigen(int n_layers, double* state, int64_t ka, int64_t kg, cudaStream_t s) {
    const int64_t nmax = ka > kg ? ka : kg;
    const int64_t mh = (nmax + 2) / 2, sq = nmax * (nmax + 1);
    const int64_t stride = (int64_t)kfac_state_bytes(ka, kg) / 8;
    cudaError_t e;
    note_launches(1);
    if (nmax <= 64) {
        const size_t smem = (size_t)3 * sq * 8 + (size_t)mh * (8 + 8) + (size_t)2 * sq * 4 + (size_t)mh * (4 + 4 + 4 + 4);
        if ((e = cudaFuncSetAttribute(jacobi_kernel<true>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem)))
            return e;
        jacobi_kernel<true><<<dim3(2, (unsigned)n_layers), kKfThreads, smem, s>>>(state, stride, ka, kg);
        return cudaGetLastError();
    }
    const size_t smem = (size_t)sq * 8 + (size_t)mh * (8 + 8 + 4 + 4);
    if ((e = cudaFuncSetAttribute(jacobi_kernel<false>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem)))
        return e;
    jacobi_kernel<false><<<dim3(2, (unsigned)n_layers), kKfThreads, smem, s>>>(state, stride, ka, kg);
    return cudaGetLastError();
}

// EK-FAC sums of n_layers layers whose features sit side by side in phi
// (layer l at column l*ka*kg); part holds n_layers * nblk * ka*kg floats.
cudaError_t launch_kfac_ekfac_accum(int n_layers, double* state, int64_t ka, int64_t kg, const float* phi, int64_t n,
                                    int64_t ld, float* part, int nblk, cudaStream_t s) {
    if (n == 0) return cudaSuccess;
    const bool su = ka <= 64 && kg <= 64;
    const size_t smem = (size_t)(2 * ka * kg + (su ? ka * ka + kg * kg : 0)) * 4;
    const int64_t stride = (int64_t)kfac_state_bytes(ka, kg) / 8;
    const dim3 grid((unsigned)nblk, (unsigned)n_layers);
    const bool aligned = ((uintptr_t)phi & 15) == 0 && (ld & 3) == 0;
    if (ka == kg && aligned && (ka == 16 || ka == 32 || ka == 64)) {
        note_launches(2);
        if (ka == 16)
            ekfac_reg_kernel<16><<<grid, 256, 0, s>>>(phi, n, ld, state, stride, part);
        else if (ka == 32)
            ekfac_reg_kernel<32><<<grid, 256, 0, s>>>(phi, n, ld, state, stride, part);
        else
            ekfac_reg_kernel<64><<<grid, 256, 0, s>>>(phi, n, ld, state, stride, part);
        ekfac_reduce_kernel<<<dim3((unsigned)((ka * kg + 255) / 256), (unsigned)n_layers), 256, 0, s>>>(
            part, nblk, state, stride, ka, kg, (double)n);
        return cudaGetLastError();
    }
    cudaError_t e = su ? cudaFuncSetAttribute(ekfac_partial_kernel<true>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                              (int)smem)
                       : cudaFuncSetAttribute(ekfac_partial_kernel<false>,
                                              cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    note_launches(2);
    if (su)
        ekfac_partial_kernel<true><<<grid, kKfThreads, smem, s>>>(phi, n, ld, state, stride, ka, kg, part);
    else
        ekfac_partial_kernel<false><<<grid, kKfThreads, smem, s>>>(phi, n, ld, state, stride, ka, kg, part);
    ekfac_reduce_kernel<<<dim3((unsigned)((ka * kg + 255) / 256), (unsigned)n_layers), 256, 0, s>>>(
        part, nblk, state, stride, ka, kg, (double)n);
    return cudaGetLastError();
}

cudaError_t launch_kfac_apply(int kind, int n_layers, const double* state, int64_t ka, int64_t kg, double lambda_abs,
                              double lambda_rel, const float* q, int64_t n_q, int64_t ld_q, float* qhat,
                              int64_t ld_qhat, cudaStream_t s) {
    if (n_q == 0) return cudaSuccess;
    const bool su = ka <= 64 && kg <= 64;
    const size_t smem = (size_t)(2 * ka * kg + (su ? ka * ka + kg * kg : 0)) * 4;
    const int64_t stride = (int64_t)kfac_state_bytes(ka, kg) / 8;
    cudaError_t e = su ? cudaFuncSetAttribute(kfac_apply_kernel<true>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                              (int)smem)
                       : cudaFuncSetAttribute(kfac_apply_kernel<false>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                              (int)smem);
    if (e != cudaSuccess) return e;
    note_launches(1);
    const dim3 grid((unsigned)n_q, (unsigned)n_layers);
    if (su)
        kfac_apply_kernel<true><<<grid, kKfThreads, smem, s>>>(kind, state, stride, ka, kg, lambda_abs, lambda_rel, q,
                                                               ld_q, qhat, ld_qhat);
    else
        kfac_apply_kernel<false><<<grid, kKfThreads, smem, s>>>(kind, state, stride, ka, kg, lambda_abs, lambda_rel,
                                                                q, ld_q, qhat, ld_qhat);
    return cudaGetLastError();
}

int64_t kfac_offset_sa(int64_t ka, int64_t kg) { return KfLayout(ka, kg).Sa; }
int64_t kfac_offset_sg(int64_t ka, int64_t kg) { return KfLayout(ka, kg).Sg; }

}  // namespace tda
