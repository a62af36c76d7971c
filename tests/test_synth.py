"""The seeded input generator: distributions, masking, offsets, bf16 rounding."""
import numpy as np
import torch

from paper_2609_38767_gb300 import synth


def test_normal_moments():
    key = synth.stream_key(1, 0)
    z = synth.normal(key, np.arange(400_000, dtype=np.uint64)).astype(np.float64)
    assert abs(z.mean()) < 4 / np.sqrt(z.size)
    assert abs(z.var() - 1.0) < 0.01
    assert np.abs(z).max() <= 6.0
    # sum of 12 uniforms: excess kurtosis -0.1 (vs 0 for a Gaussian)
    k = ((z - z.mean()) ** 4).mean() / z.var() ** 2 - 3
    assert -0.16 < k < -0.04


def test_student_t4_is_heavy_tailed():
    key = synth.stream_key(1, 5)
    t = synth.student_t4(key, np.arange(200_000, dtype=np.uint64)).astype(np.float64)
    assert abs(np.median(t)) < 0.02
    # t_4: variance nu/(nu-2) = 2; P(|t| > 4.604) = 0.01
    assert 1.7 < t.var() < 2.4
    assert 0.007 < (np.abs(t) > 4.604).mean() < 0.013


def test_offsets_and_streams_are_consistent():
    full = synth.factors(2, 3, 7, 5, 24, sigma=0.5, dtype="f32")
    part = synth.factors(2, 3, 2, 5, 24, sigma=0.5, e0=5, dtype="f32")
    np.testing.assert_array_equal(full[5:7], part)
    other = synth.factors(2, 4, 7, 5, 24, sigma=0.5, dtype="f32")
    assert not np.array_equal(full, other)


def test_mask_zeroes_whole_tokens_at_rate_p():
    A = synth.factors(1, 0, 64, 256, 8, dtype="f32", mask_p=0.01)
    B = synth.factors(2, 0, 64, 256, 16, dtype="f32", mask_p=0.01)
    za = np.all(A == 0, axis=2)
    zb = np.all(B == 0, axis=2)
    assert np.array_equal(za, zb)  # same tokens masked in both factors
    frac = za.mean()
    assert abs(frac - 0.01) < 4 * np.sqrt(0.01 * 0.99 / za.size)


def test_bf16_rounding_matches_torch():
    x = synth.factors(1, 9, 3, 17, 40, sigma=0.1, dtype="f32")
    bits = synth.f32_to_bf16_bits(x)
    ref = torch.from_numpy(x).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    np.testing.assert_array_equal(bits, ref)
    np.testing.assert_array_equal(synth.factors(1, 9, 3, 17, 40, sigma=0.1, dtype="bf16"), bits)


def test_sigma_scales_in_fp32():
    a = synth.factors(1, 0, 2, 3, 8, sigma=1.0, dtype="f32")
    b = synth.factors(1, 0, 2, 3, 8, sigma=0.1, dtype="f32")
    np.testing.assert_array_equal(b, (a * np.float32(0.1)).astype(np.float32))


def test_c_generator_matches_numpy_definition():
    from paper_2609_38767_gb300 import build

    build.build_synth_cpu()
    for dtype, dist, mask in [("f32", 0, 0.0), ("bf16", 0, 0.01), ("bf16", 1, 0.0), ("f32", 1, 0.05)]:
        a = synth.factors(5, 7, 3, 37, 48, 0.37, dist, 11, dtype, mask, impl="numpy")
        b = synth.factors(5, 7, 3, 37, 48, 0.37, dist, 11, dtype, mask, impl="c")
        np.testing.assert_array_equal(a, b)
