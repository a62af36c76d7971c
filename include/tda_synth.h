/*
 * tda_synth.h -- C ABI of libtda_synth.so, the seeded synthetic-factor
 * generator used by the tests and the benchmark to create device-resident
 * inputs. It is NOT a step of the attribution method: it only fills buffers
 * with the values defined in paper_2609_38767_gb300/synth.py (same bits as
 * that numpy implementation, so sampled examples can be regenerated on the
 * CPU for the oracle).
 */
#ifndef TDA_SYNTH_H
#define TDA_SYNTH_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* Fill X[n][T][d] (device; dtype 0 = fp32, 1 = bf16) with
 * dist(key(seed, stream), i) * sigma, i = ((e0 + n)*T + t)*d + c, dist 0 =
 * sum-of-twelve-uniforms normal, 1 = Student-t with 4 degrees of freedom.
 * Tokens with word(key(mask_seed, mask_stream), e*T + t) < mask_threshold are
 * zero (mask_threshold 0 disables masking). Asynchronous on `stream`.
 * Returns 0 on success, 1 on a bad argument, 2 on a CUDA error. */
int32_t tda_synth_fill(void* X, int32_t dtype, int32_t dist, uint64_t seed, uint64_t stream_id,
                       int64_t e0, int64_t n, int64_t T, int64_t d, float sigma,
                       uint64_t mask_seed, uint64_t mask_stream, uint64_t mask_threshold,
                       void* stream);

#ifdef __cplusplus
}
#endif
#endif /* TDA_SYNTH_H */
