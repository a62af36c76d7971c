// k_project_simt.cu -- sign-matrix dump and the generic (CUDA-core) factored
// projection, for any layer shape, fp32 or bf16 factors.
//
// Factored projection, Eq. 2: for every example n,
//   At = A_n S_in (T x k_in), Bt = B_n S_out (T x k_out),
//   Phi_n = scale * Bt^T At (k_out x k_in), scale = 1/sqrt(k_in k_out),
// with S generated on chip from the counter hash (App. A.2) and never stored.
// This kernel is the fp32 path (its 1e-5 tolerance excludes TF32 tensor
// cores) and the fallback for shapes the tensor-core kernel does not cover.
#include <cuda_bf16.h>

#include "tda_internal.cuh"

namespace tda {
namespace {

constexpr int kTile = 64;      // Phi tile edge: rows i (k_out), columns j (k_in)
constexpr int kTokChunk = 16;  // tokens per contraction step
constexpr int kDChunk = 64;    // rows of S per sign word
constexpr int kThreads = 256;

__device__ __forceinline__ float load_elem(const float* p) { return __ldg(p); }
__device__ __forceinline__ float load_elem(const __nv_bfloat16* p) { return __bfloat162float(*p); }

__global__ void proj_entries_kernel(uint64_t key, int kind, int64_t rows, int32_t cols,
                                    int8_t* __restrict__ out) {
    const int64_t total = rows * (int64_t)cols;
    for (int64_t e = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; e < total;
         e += (int64_t)gridDim.x * blockDim.x) {
        const int64_t r = e / cols;
        const int32_t c = (int32_t)(e - r * cols);
        int8_t v;
        if (kind == TDA_PROJ_IDENTITY)
            v = (r == c) ? 1 : 0;
        else
            v = ((sign_word(key, (uint32_t)c, (uint64_t)(r >> 6)) >> (r & 63)) & 1u) ? -1 : 1;
        out[e] = v;
    }
}

// X[t][j] = sum_c src[t0+t][c] * S[c][c0+j] for a chunk of kTokChunk tokens
// and a kTile-wide column tile. Thread (t = tid/16, 4 columns at (tid%16)*4).
template <typename T>
__device__ __forceinline__ void project_chunk(const T* __restrict__ src, int64_t Tn, int64_t d,
                                              int64_t t0, uint64_t key, int kind, int c0,
                                              float (*Xs)[kTile], float (*Vs)[kDChunk + 1],
                                              uint64_t* Ws) {
    const int tid = threadIdx.x;
    const int t = tid / 16, jq = (tid % 16) * 4;
    float o[4] = {0.f, 0.f, 0.f, 0.f};
    for (int64_t dc = 0; dc < d; dc += kDChunk) {
        __syncthreads();  // previous readers of Vs / Ws are done
        for (int e = tid; e < kTokChunk * kDChunk; e += kThreads) {
            const int tt = e / kDChunk, cc = e % kDChunk;
            const int64_t tg = t0 + tt, cg = dc + cc;
            Vs[tt][cc] = (tg < Tn && cg < d) ? load_elem(src + tg * d + cg) : 0.f;
        }
        if (kind == TDA_PROJ_RADEMACHER && tid < kTile)
            Ws[tid] = sign_word(key, (uint32_t)(c0 + tid), (uint64_t)(dc >> 6));
        __syncthreads();
        if (kind == TDA_PROJ_RADEMACHER) {
            const uint64_t w0 = Ws[jq], w1 = Ws[jq + 1], w2 = Ws[jq + 2], w3 = Ws[jq + 3];
#pragma unroll 8
            for (int r = 0; r < kDChunk; ++r) {
                const float v = Vs[t][r];
                o[0] += ((w0 >> r) & 1u) ? -v : v;
                o[1] += ((w1 >> r) & 1u) ? -v : v;
                o[2] += ((w2 >> r) & 1u) ? -v : v;
                o[3] += ((w3 >> r) & 1u) ? -v : v;
            }
        } else {  // identity map: S[c][j] = [c == j]
#pragma unroll
            for (int q = 0; q < 4; ++q) {
                const int64_t jg = c0 + jq + q;
                if (jg >= dc && jg < dc + kDChunk) o[q] += Vs[t][jg - dc];
            }
        }
    }
#pragma unroll
    for (int q = 0; q < 4; ++q) Xs[t][jq + q] = o[q];
}

template <typename T>
__global__ void __launch_bounds__(kThreads)
project_simt_kernel(const T* __restrict__ A, const T* __restrict__ B, int64_t Tn, int64_t d_in,
                    int64_t d_out, int k_in, int k_out, uint64_t key_in, uint64_t key_out,
                    int kind, float scale, float* __restrict__ phi, int64_t ld_phi) {
    __shared__ float Xs[kTokChunk][kTile];       // At chunk, column tile j0
    __shared__ float Ys[kTokChunk][kTile];       // Bt chunk, column tile i0
    __shared__ float Vs[kTokChunk][kDChunk + 1]; // staged factor rows
    __shared__ uint64_t Ws[kTile];               // sign words of the current 64-row block

    const int64_t n = blockIdx.x;
    const int i0 = blockIdx.y * kTile;
    const int j0 = blockIdx.z * kTile;
    const T* An = A + n * Tn * d_in;
    const T* Bn = B + n * Tn * d_out;
    const int tid = threadIdx.x;
    const int ri = (tid / 16) * 4, cj = (tid % 16) * 4;
    float acc[4][4];
#pragma unroll
    for (int a = 0; a < 4; ++a)
#pragma unroll
        for (int b = 0; b < 4; ++b) acc[a][b] = 0.f;

    for (int64_t t0 = 0; t0 < Tn; t0 += kTokChunk) {
        project_chunk(An, Tn, d_in, t0, key_in, kind, j0, Xs, Vs, Ws);
        project_chunk(Bn, Tn, d_out, t0, key_out, kind, i0, Ys, Vs, Ws);
        __syncthreads();
#pragma unroll 4
        for (int t = 0; t < kTokChunk; ++t) {
            float y[4], x[4];
#pragma unroll
            for (int a = 0; a < 4; ++a) y[a] = Ys[t][ri + a];
#pragma unroll
            for (int b = 0; b < 4; ++b) x[b] = Xs[t][cj + b];
#pragma unroll
            for (int a = 0; a < 4; ++a)
#pragma unroll
                for (int b = 0; b < 4; ++b) acc[a][b] = fmaf(y[a], x[b], acc[a][b]);
        }
        __syncthreads();
    }
#pragma unroll
    for (int a = 0; a < 4; ++a)
#pragma unroll
        for (int b = 0; b < 4; ++b) {
            const int i = i0 + ri + a, j = j0 + cj + b;
            if (i < k_out && j < k_in) phi[n * ld_phi + (int64_t)i * k_in + j] = acc[a][b] * scale;
        }
}

}  // namespace

cudaError_t launch_proj_entries(uint64_t key, int kind, int64_t rows, int32_t cols, int8_t* out,
                                cudaStream_t s) {
    const int64_t total = rows * (int64_t)cols;
    if (total == 0) return cudaSuccess;
    int64_t blocks = (total + 255) / 256;
    if (blocks > 152 * 64) blocks = 152 * 64;
    note_launches(1);
    proj_entries_kernel<<<(unsigned)blocks, 256, 0, s>>>(key, kind, rows, cols, out);
    return cudaGetLastError();
}

float projection_scale(const tda_layer_desc& L) {
    if (L.kind == TDA_PROJ_IDENTITY) return 1.0f;
    return (float)(1.0 / (sqrt((double)L.k_in) * sqrt((double)L.k_out)));
}

cudaError_t launch_project_simt(const tda_layer_desc& L, tda_dtype dt, const void* A, const void* B,
                                int64_t N, float* phi, int64_t ld_phi, cudaStream_t s) {
    if (N == 0) return cudaSuccess;
    const uint64_t key_in = side_key(L.seed, L.layer, 0);
    const uint64_t key_out = side_key(L.seed, L.layer, 1);
    dim3 grid((unsigned)N, (unsigned)((L.k_out + kTile - 1) / kTile),
              (unsigned)((L.k_in + kTile - 1) / kTile));
    const float scale = projection_scale(L);
    note_launches(1);
    if (dt == TDA_BF16)
        project_simt_kernel<__nv_bfloat16><<<grid, kThreads, 0, s>>>(
            (const __nv_bfloat16*)A, (const __nv_bfloat16*)B, L.T, L.d_in, L.d_out, L.k_in,
            L.k_out, key_in, key_out, L.kind, scale, phi, ld_phi);
    else
        project_simt_kernel<float><<<grid, kThreads, 0, s>>>(
            (const float*)A, (const float*)B, L.T, L.d_in, L.d_out, L.k_in, L.k_out, key_in,
            key_out, L.kind, scale, phi, ld_phi);
    return cudaGetLastError();
}

}  // namespace tda
