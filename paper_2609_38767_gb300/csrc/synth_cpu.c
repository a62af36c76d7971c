/* synth_cpu.c -- CPU implementation of the seeded synthetic-factor generator
 * (libtda_synth_cpu.so). Same definition, and the same bits, as the numpy
 * version in paper_2609_38767_gb300/synth.py and the device version in
 * synth.cu; it exists because regenerating full-size sampled examples in numpy
 * is slow. Built with -ffp-contract=off so every fp32 operation rounds once. */
#include <math.h>
#include <stdint.h>
#include <string.h>

#define G 0x9E3779B97F4A7C15ULL

static uint64_t smix(uint64_t z) {
    z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ULL;
    z = (z ^ (z >> 27)) * 0x94D049BB133111EBULL;
    return z ^ (z >> 31);
}
static uint64_t sword(uint64_t key, uint64_t n) { return smix(key + G * (n + 1u)); }

static float snormal(uint64_t key, uint64_t i) {
    int64_t s = 0;
    for (int j = 0; j < 3; ++j) {
        uint64_t w = sword(key, 3u * i + (uint64_t)j);
        s += (int64_t)(w & 0xFFFFu) + (int64_t)((w >> 16) & 0xFFFFu) + (int64_t)((w >> 32) & 0xFFFFu) +
             (int64_t)((w >> 48) & 0xFFFFu);
    }
    return (float)(s + 6 - 393216) / 65536.0f;
}

static float sstudent4(uint64_t key, uint64_t i) {
    uint64_t b = 5u * i;
    float z0 = snormal(key, b), z1 = snormal(key, b + 1), z2 = snormal(key, b + 2), z3 = snormal(key, b + 3),
          z4 = snormal(key, b + 4);
    float s = z1 * z1;
    s = s + z2 * z2;
    s = s + z3 * z3;
    s = s + z4 * z4;
    s = s * 0.25f;
    return s > 0.f ? z0 / sqrtf(s) : 0.f;
}

static uint16_t to_bf16(float v) {
    uint32_t u;
    memcpy(&u, &v, 4);
    return (uint16_t)((u + ((u >> 16) & 1u) + 0x7FFFu) >> 16);
}

/* X[n][T][d], dtype 0 = fp32, 1 = bf16 bits. Returns 0, or 1 on a bad argument. */
int32_t tda_synth_fill_cpu(void* X, int32_t dtype, int32_t dist, uint64_t seed, uint64_t stream_id, int64_t e0,
                           int64_t n, int64_t T, int64_t d, float sigma, uint64_t mask_seed, uint64_t mask_stream,
                           uint64_t mask_threshold) {
    if ((dtype != 0 && dtype != 1) || (dist != 0 && dist != 1) || n < 0 || T < 0 || d < 0 || e0 < 0) return 1;
    const uint64_t key = smix(seed + G * (stream_id + 1u));
    const uint64_t mkey = smix(mask_seed + G * (mask_stream + 1u));
    const int64_t rows = n * T;
#pragma omp parallel for schedule(static)
    for (int64_t r = 0; r < rows; ++r) {
        const int64_t ex = r / T, t = r - ex * T;
        const uint64_t tok = (uint64_t)(e0 + ex) * (uint64_t)T + (uint64_t)t;
        const int keep = mask_threshold == 0 || sword(mkey, tok) >= mask_threshold;
        for (int64_t c = 0; c < d; ++c) {
            float v = 0.f;
            if (keep) {
                const uint64_t i = tok * (uint64_t)d + (uint64_t)c;
                v = (dist == 0 ? snormal(key, i) : sstudent4(key, i)) * sigma;
            }
            if (dtype == 1)
                ((uint16_t*)X)[r * d + c] = to_bf16(v);
            else
                ((float*)X)[r * d + c] = v;
        }
    }
    return 0;
}
