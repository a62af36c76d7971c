// k_score.cu -- score GEMM S = beta*S + Qhat Phi^T (gradient inner products,
// Sec. 3.2 / Eq. 4's left side; GradDot when Qhat = Q) and per-row top-k.
#include <float.h>

#include "tda_internal.cuh"

namespace tda {
namespace {

constexpr int kTQ = 32;   // queries per tile
constexpr int kTT = 64;   // train examples per tile
constexpr int kSK = 32;   // feature chunk
constexpr int kSThreads = 256;

__device__ __forceinline__ void load4(const float* p, bool ok, bool vec, float* out, int64_t lim) {
    if (ok && vec) {
        const float4 v = *reinterpret_cast<const float4*>(p);
        out[0] = v.x; out[1] = v.y; out[2] = v.z; out[3] = v.w;
    } else {
        for (int i = 0; i < 4; ++i) out[i] = (ok && i < lim) ? p[i] : 0.f;
    }
}
__device__ __forceinline__ void load4(const double* p, bool ok, bool, double* out, int64_t lim) {
    for (int i = 0; i < 4; ++i) out[i] = (ok && i < lim) ? p[i] : 0.0;
}

// S tile (32 queries x 64 train) = Qhat_tile Phi_tile^T over D in chunks of 32.
// Thread (tq = tid/32, tt = tid%32) owns queries tq*4..+3 and train tt, tt+32.
// Operands are read 16 bytes at a time along the feature axis (coalesced) and
// staged transposed ([feature][row], padded) in shared memory.
template <typename TQ, typename TA>
__global__ void __launch_bounds__(kSThreads)
score_kernel(const TQ* __restrict__ Q, int64_t n_q, int64_t ld_q, const float* __restrict__ P,
             int64_t n_t, int64_t ld_p, int64_t D, float* __restrict__ S, int64_t ld_S,
             float beta, int64_t kslice, int64_t slab) {
    __shared__ TA Qs[kSK][kTQ + 1];
    __shared__ TA Ps[kSK][kTT + 1];
    const int tid = threadIdx.x;
    {   // split K: slice blockIdx.z of the features into its own slab of S
        const int64_t k0 = (int64_t)blockIdx.z * kslice;
        Q += k0;
        P += k0;
        D = D - k0 < kslice ? D - k0 : kslice;
        S += (int64_t)blockIdx.z * slab;
    }
    const int64_t q0 = (int64_t)blockIdx.y * kTQ, i0 = (int64_t)blockIdx.x * kTT;
    const int tq = tid >> 5, tt = tid & 31;
    const bool vq = (sizeof(TQ) == 4) && ((ld_q & 3) == 0) && (((uintptr_t)Q & 15) == 0);
    const bool vp = ((ld_p & 3) == 0) && (((uintptr_t)P & 15) == 0);
    TA acc[4][2];
#pragma unroll
    for (int a = 0; a < 4; ++a) acc[a][0] = acc[a][1] = (TA)0;

    for (int64_t f0 = 0; f0 < D; f0 += kSK) {
        {   // Q tile: 32 rows x 32 features, one 4-wide load per thread
            const int r = tid >> 3, k4 = (tid & 7) * 4;
            const int64_t q = q0 + r, f = f0 + k4;
            TQ v[4];
            load4(Q + q * ld_q + f, q < n_q && f < D, vq && f + 3 < D, v, D - f);
#pragma unroll
            for (int i = 0; i < 4; ++i) Qs[k4 + i][r] = (TA)v[i];
        }
#pragma unroll
        for (int h = 0; h < 2; ++h) {  // Phi tile: 64 rows x 32 features
            const int e = tid + h * kSThreads;
            const int r = e >> 3, k4 = (e & 7) * 4;
            const int64_t i = i0 + r, f = f0 + k4;
            float v[4];
            load4(P + i * ld_p + f, i < n_t && f < D, vp && f + 3 < D, v, D - f);
#pragma unroll
            for (int u = 0; u < 4; ++u) Ps[k4 + u][r] = (TA)v[u];
        }
        __syncthreads();
#pragma unroll 8
        for (int k = 0; k < kSK; ++k) {
            TA a[4];
#pragma unroll
            for (int u = 0; u < 4; ++u) a[u] = Qs[k][tq * 4 + u];
            const TA b0 = Ps[k][tt], b1 = Ps[k][tt + 32];
#pragma unroll
            for (int u = 0; u < 4; ++u) {
                acc[u][0] += a[u] * b0;
                acc[u][1] += a[u] * b1;
            }
        }
        __syncthreads();
    }
#pragma unroll
    for (int u = 0; u < 4; ++u)
#pragma unroll
        for (int v = 0; v < 2; ++v) {
            const int64_t q = q0 + tq * 4 + u, i = i0 + tt + 32 * v;
            if (q < n_q && i < n_t) {
                float* dst = S + q * ld_S + i;
                *dst = (beta == 0.f) ? (float)acc[u][v] : (float)((TA)beta * (TA)(*dst) + acc[u][v]);
            }
        }
}

// ---------------------------------------------------------------------------
// Top-k. Each entry gets a 64-bit key whose descending order is "score
// descending, then index ascending": the high word maps the float to an
// order-preserving unsigned (NaN largest, -0 folded into +0), the low word is
// ~index. Keys are distinct, so the k-th largest key splits the row exactly.
// One CTA per row: 8 passes of an 8-bit radix select find that key, the k
// winners are gathered and bitonic-sorted in shared memory.
// ---------------------------------------------------------------------------
constexpr int kTopThreads = 512;
constexpr int kTopMaxK = 1024;

__device__ __forceinline__ uint64_t topk_key(float v, int64_t i) {
    uint32_t u = __float_as_uint(v);
    uint32_t o;
    if (v != v)
        o = 0xFFFFFFFFu;
    else if (v == 0.f)
        o = 0x80000000u;
    else
        o = (u & 0x80000000u) ? ~u : (u | 0x80000000u);
    return ((uint64_t)o << 32) | (uint64_t)(~(uint32_t)i);
}

__global__ void __launch_bounds__(kTopThreads)
topk_kernel(const float* __restrict__ S, int64_t n_t, int64_t ld_S, int32_t k,
            int32_t* __restrict__ idx, float* __restrict__ val) {
    __shared__ unsigned int hist[256];
    __shared__ uint64_t sel[kTopMaxK];
    __shared__ uint64_t s_prefix, s_mask;
    __shared__ int s_remaining;
    __shared__ unsigned int s_count;
    const int64_t q = blockIdx.x;
    const float* row = S + q * ld_S;
    const int tid = threadIdx.x;
    if (tid == 0) {
        s_prefix = 0;
        s_mask = 0;
        s_remaining = k;
        s_count = 0;
    }
    for (int pass = 0; pass < 8; ++pass) {
        const int shift = 56 - 8 * pass;
        for (int b = tid; b < 256; b += kTopThreads) hist[b] = 0;
        __syncthreads();
        const uint64_t prefix = s_prefix, mask = s_mask;
        for (int64_t i = tid; i < n_t; i += kTopThreads) {
            const uint64_t key = topk_key(row[i], i);
            if ((key & mask) == prefix) atomicAdd(&hist[(key >> shift) & 255u], 1u);
        }
        __syncthreads();
        if (tid == 0) {
            int rem = s_remaining;
            unsigned int cum = 0;
            int digit = 0;
            for (int b = 255; b >= 0; --b) {
                if (cum + hist[b] >= (unsigned)rem) {
                    digit = b;
                    break;
                }
                cum += hist[b];
            }
            s_remaining = rem - (int)cum;
            s_prefix = prefix | ((uint64_t)digit << shift);
            s_mask = mask | ((uint64_t)255 << shift);
        }
        __syncthreads();
    }
    const uint64_t kth = s_prefix;  // the k-th largest key
    int P = 1;
    while (P < k) P <<= 1;
    for (int e = tid; e < P; e += kTopThreads) sel[e] = 0;
    __syncthreads();
    for (int64_t i = tid; i < n_t; i += kTopThreads) {
        const uint64_t key = topk_key(row[i], i);
        if (key >= kth) {
            const unsigned int slot = atomicAdd(&s_count, 1u);
            if (slot < (unsigned)k) sel[slot] = key;
        }
    }
    __syncthreads();
    // bitonic sort, descending
    for (int size = 2; size <= P; size <<= 1) {
        for (int stride = size >> 1; stride > 0; stride >>= 1) {
            for (int e = tid; e < P; e += kTopThreads) {
                const int partner = e ^ stride;
                if (partner > e) {
                    const bool desc = ((e & size) == 0);
                    const uint64_t a = sel[e], b = sel[partner];
                    if (desc ? (a < b) : (a > b)) {
                        sel[e] = b;
                        sel[partner] = a;
                    }
                }
            }
            __syncthreads();
        }
    }
    for (int e = tid; e < k; e += kTopThreads) {
        const uint32_t i = ~(uint32_t)(sel[e] & 0xFFFFFFFFu);
        const bool ok = (int64_t)i < n_t;  // always true when exactly k keys were selected
        idx[q * k + e] = ok ? (int32_t)i : -1;
        if (val) val[q * k + e] = ok ? row[i] : __int_as_float(0x7fc00000);
    }
}

}  // namespace

cudaError_t launch_score(const void* Qhat, tda_dtype qdt, int64_t n_q, int64_t ld_q,
                         const float* Phi, int64_t n_t, int64_t ld_phi, int64_t D, float* S,
                         int64_t ld_S, float beta, cudaStream_t s) {
    if (n_q == 0 || n_t == 0) return cudaSuccess;
    dim3 grid((unsigned)((n_t + kTT - 1) / kTT), (unsigned)((n_q + kTQ - 1) / kTQ));
    note_launches(1);
    if (qdt == TDA_F64)
        score_kernel<double, double><<<grid, kSThreads, 0, s>>>(
            (const double*)Qhat, n_q, ld_q, Phi, n_t, ld_phi, D, S, ld_S, beta, D, 0);
    else
        score_kernel<float, float><<<grid, kSThreads, 0, s>>>(
            (const float*)Qhat, n_q, ld_q, Phi, n_t, ld_phi, D, S, ld_S, beta, D, 0);
    return cudaGetLastError();
}

namespace {
// S[q][i] = beta * S[q][i] + sum_z part[z][q][i] (slabs of n_q x n_t, fixed order)
__global__ void sum_slabs_kernel(const float* __restrict__ part, int splits, int64_t n_q, int64_t n_t,
                                 float* __restrict__ S, int64_t ld_S, float beta) {
    const int64_t total = n_q * n_t;
    for (int64_t e = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; e < total; e += (int64_t)gridDim.x * blockDim.x) {
        float v = 0.f;
        for (int z = 0; z < splits; ++z) v += part[z * total + e];
        const int64_t q = e / n_t, i = e - q * n_t;
        float* dst = S + q * ld_S + i;
        *dst = beta == 0.f ? v : beta * (*dst) + v;
    }
}
}  // namespace

bool score_dots_tc(const float* Q, int64_t n_q, int64_t ld_q, const float* Phi, int64_t n_t, int64_t ld_phi,
                   int64_t D) {
    return device_error_word() != nullptr && score_tc_supported(TDA_F32, Q, n_q, ld_q, Phi, n_t, ld_phi, D);
}

int score_splitk_splits(int64_t n_q, int64_t n_t, int64_t D, bool tc) {
    int64_t z;
    if (tc) {
        // one 3xTF32 CTA per SM (about 200 KiB of shared memory each), slices of >= 4096 features
        static int sms = 0;
        if (!sms) {
            int dev = 0;
            cudaGetDevice(&dev);
            cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
            if (sms <= 0) sms = 1;
        }
        const int64_t tiles = score_tc_tiles(n_q, n_t);
        z = sms / (tiles > 0 ? tiles : 1);
        if (z > D / 4096) z = D / 4096;
    } else {
        const int64_t tiles = ((n_t + kTT - 1) / kTT) * ((n_q + kTQ - 1) / kTQ);
        z = 608 / (tiles > 0 ? tiles : 1);
        if (z > D / 1024) z = D / 1024;  // at least 1024 features per slice
    }
    if (z > 256) z = 256;
    return z < 2 ? 1 : (int)z;
}

// fp32 score with the feature axis split over `splits` CTAs per tile: for
// few, very long rows (inner products of materialised gradients). part: device
// scratch of splits * n_q * n_t floats. tc: the 3xTF32 tensor-core kernel
// (score_dots_tc said yes), else the CUDA-core one.
cudaError_t launch_score_splitk(const float* Q, int64_t n_q, int64_t ld_q, const float* Phi, int64_t n_t,
                                int64_t ld_phi, int64_t D, float* S, int64_t ld_S, float beta, int splits,
                                float* part, bool tc, cudaStream_t s) {
    if (n_q == 0 || n_t == 0) return cudaSuccess;
    if (tc) {
        unsigned int* err = device_error_word();
        if (splits <= 1) return launch_score_tc(Q, n_q, ld_q, Phi, n_t, ld_phi, D, S, ld_S, beta, err, s);
        int64_t kslice = (D + splits - 1) / splits;
        kslice = (kslice + 31) / 32 * 32;
        const int z = (int)((D + kslice - 1) / kslice);
        cudaError_t e = launch_score_tc_slices(Q, n_q, ld_q, Phi, n_t, ld_phi, D, splits, part, err, s);
        if (e != cudaSuccess) return e;
        int64_t blocks = (n_q * n_t + 255) / 256;
        if (blocks > 4096) blocks = 4096;
        note_launches(1);
        sum_slabs_kernel<<<(unsigned)blocks, 256, 0, s>>>(part, z, n_q, n_t, S, ld_S, beta);
        return cudaGetLastError();
    }
    if (splits <= 1) return launch_score(Q, TDA_F32, n_q, ld_q, Phi, n_t, ld_phi, D, S, ld_S, beta, s);
    int64_t kslice = (D + splits - 1) / splits;
    kslice = (kslice + kSK - 1) / kSK * kSK;
    const int z = (int)((D + kslice - 1) / kslice);
    dim3 grid((unsigned)((n_t + kTT - 1) / kTT), (unsigned)((n_q + kTQ - 1) / kTQ), (unsigned)z);
    note_launches(2);
    score_kernel<float, float><<<grid, kSThreads, 0, s>>>(Q, n_q, ld_q, Phi, n_t, ld_phi, D, part, n_t, 0.f, kslice,
                                                          n_q * n_t);
    int64_t blocks = (n_q * n_t + 255) / 256;
    if (blocks > 4096) blocks = 4096;
    sum_slabs_kernel<<<(unsigned)blocks, 256, 0, s>>>(part, z, n_q, n_t, S, ld_S, beta);
    return cudaGetLastError();
}

cudaError_t launch_topk(const float* S, int64_t n_q, int64_t n_t, int64_t ld_S, int32_t k,
                        int32_t* idx, float* val, cudaStream_t s) {
    if (n_q == 0) return cudaSuccess;
    note_launches(1);
    topk_kernel<<<(unsigned)n_q, kTopThreads, 0, s>>>(S, n_t, ld_S, k, idx, val);
    return cudaGetLastError();
}

}  // namespace tda
