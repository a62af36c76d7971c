"""Seeded synthetic factor generator (inputs only; none of the method's arithmetic).

Both the CPU oracle and the CUDA library consume inputs from this one
definition. It is implemented twice, bit-identically: here in numpy (for the
oracle and for small test inputs) and in ``csrc/synth.cu`` (``libtda_synth.so``,
for device-resident inputs at full size). A value depends only on
(seed, stream, global element index), so any sampled subset of a full-size
device tensor can be regenerated on the CPU without reading it back.

Definition (all integer arithmetic mod 2^64, floating point in IEEE fp32 with
one rounding per operation):

* ``mix64`` is the SplitMix64 output function (Steele, Lea & Flood 2014);
  ``key(seed, stream) = mix64(seed + G*(stream+1))`` and
  ``word(key, n) = mix64(key + G*(n+1))`` with G = 0x9E3779B97F4A7C15.
* ``normal(key, i)``: the twelve 16-bit fields x_0..x_11 of
  word(key, 3i), word(key, 3i+1), word(key, 3i+2) give
  z = (sum x_j + 6 - 393216) / 65536 = sum_j u_j - 6 with u_j = (x_j + 1/2)/2^16,
  the classical sum-of-twelve-uniforms approximation of N(0, 1): mean 0,
  variance exactly 1, support [-6, 6]. Exact in fp32.
* ``student_t4(key, i)``: with z_j = normal(key, 5i+j),
  s = (((z1*z1 + z2*z2) + z3*z3) + z4*z4) * 0.25 and t = z0 / sqrt(s)
  (t = 0 if s == 0): Student-t with 4 degrees of freedom.
* An element of X[n][t][c] (n counted from example offset e0, T tokens,
  width d) has index i = ((e0+n)*T + t)*d + c and value dist(key, i) * sigma
  (sigma a float32), rounded to bfloat16 (round to nearest even) for bf16.
* Token masking: token (e, t) is zeroed in every factor of example e when
  word(mask_key, e*T + t) < mask_threshold, mask_threshold = floor(p * 2^64).
"""
from __future__ import annotations

import os

import numpy as np

GAMMA = np.uint64(0x9E3779B97F4A7C15)
_C1 = np.uint64(0xBF58476D1CE4E5B9)
_C2 = np.uint64(0x94D049BB133111EB)

DIST_NORMAL = 0
DIST_STUDENT_T4 = 1

# Seeds of the factor roles; queries use stream + QUERY_STREAM_OFFSET.
SEED_A = 1
SEED_B = 2
SEED_MASK = 3
QUERY_STREAM_OFFSET = 1000


def mix64(z: np.ndarray) -> np.ndarray:
    z = np.asarray(z, dtype=np.uint64)
    with np.errstate(over="ignore"):
        z = (z ^ (z >> np.uint64(30))) * _C1
        z = (z ^ (z >> np.uint64(27))) * _C2
    return z ^ (z >> np.uint64(31))


def stream_key(seed: int, stream: int) -> np.uint64:
    with np.errstate(over="ignore"):
        return mix64(np.uint64(seed) + GAMMA * np.uint64(stream + 1))[()]


def word(key: np.uint64, n: np.ndarray) -> np.ndarray:
    with np.errstate(over="ignore"):
        return mix64(np.uint64(key) + GAMMA * (np.asarray(n, dtype=np.uint64) + np.uint64(1)))


_PAIR = np.uint64(0x0000FFFF0000FFFF)
_LO32 = np.uint64(0xFFFFFFFF)


def normal(key: np.uint64, i: np.ndarray) -> np.ndarray:
    i = np.asarray(i, dtype=np.uint64)
    s = np.zeros(i.shape, dtype=np.uint64)
    with np.errstate(over="ignore"):
        base = i * np.uint64(3)
        for j in range(3):
            w = word(key, base + np.uint64(j))
            # sum of the four 16-bit fields: pairwise in two 32-bit lanes, then the lanes
            p = (w & _PAIR) + ((w >> np.uint64(16)) & _PAIR)
            s += (p & _LO32) + (p >> np.uint64(32))
    return (s.astype(np.int64) + (6 - 393216)).astype(np.float32) / np.float32(65536.0)


def student_t4(key: np.uint64, i: np.ndarray) -> np.ndarray:
    i = np.asarray(i, dtype=np.uint64)
    with np.errstate(over="ignore"):
        base = i * np.uint64(5)
    z = [normal(key, base + np.uint64(j)) for j in range(5)]
    s = z[1] * z[1]
    s = s + z[2] * z[2]
    s = s + z[3] * z[3]
    s = s + z[4] * z[4]
    s = s * np.float32(0.25)
    with np.errstate(divide="ignore", invalid="ignore"):
        t = z[0] / np.sqrt(s)
    return np.where(s > 0, t, np.float32(0.0)).astype(np.float32)


def f32_to_bf16_bits(x: np.ndarray) -> np.ndarray:
    """Round-to-nearest-even fp32 -> bf16, returned as uint16 bit patterns (finite inputs)."""
    u = np.ascontiguousarray(x, dtype=np.float32).view(np.uint32).astype(np.uint64)
    bias = ((u >> np.uint64(16)) & np.uint64(1)) + np.uint64(0x7FFF)
    return ((u + bias) >> np.uint64(16)).astype(np.uint16)


def bf16_bits_to_f32(b: np.ndarray) -> np.ndarray:
    return (np.asarray(b, dtype=np.uint16).astype(np.uint32) << np.uint32(16)).view(np.float32)


def mask_threshold(p: float) -> int:
    """floor(p * 2^64) computed from the double p, the integer both generators use."""
    if p <= 0.0:
        return 0
    return min(int(float(p) * 18446744073709551616.0), (1 << 64) - 1)


_cpu_lib = None


def _load_cpu_lib():
    """The C implementation of this generator (libtda_synth_cpu.so), or None if not built."""
    global _cpu_lib
    if _cpu_lib is None:
        import ctypes

        path = os.path.join(os.path.dirname(os.path.abspath(__file__)), "libtda_synth_cpu.so")
        if not os.path.exists(path):
            return None
        lib = ctypes.CDLL(path)
        u64, i64, i32 = ctypes.c_uint64, ctypes.c_int64, ctypes.c_int32
        lib.tda_synth_fill_cpu.restype = i32
        lib.tda_synth_fill_cpu.argtypes = [ctypes.c_void_p, i32, i32, u64, u64, i64, i64, i64, i64,
                                           ctypes.c_float, u64, u64, u64]
        _cpu_lib = lib
    return _cpu_lib


def factors(seed: int, stream: int, n: int, T: int, d: int, sigma: float = 1.0,
            dist: int = DIST_NORMAL, e0: int = 0, dtype: str = "bf16",
            mask_p: float = 0.0, mask_seed: int = SEED_MASK, mask_stream: int = 0,
            impl: str = "auto") -> np.ndarray:
    """X[n][T][d] as float32, or as uint16 bf16 bit patterns when dtype == 'bf16'.

    impl 'numpy' evaluates the definition with numpy; 'c' (or 'auto' when the
    library is built) uses the identical C implementation, which is faster."""
    lib = _load_cpu_lib() if impl in ("auto", "c") else None
    if impl == "c" and lib is None:
        raise ImportError("libtda_synth_cpu.so is not built")
    if lib is not None:
        out = np.empty((n, T, d), dtype=np.uint16 if dtype == "bf16" else np.float32)
        rc = lib.tda_synth_fill_cpu(out.ctypes.data, 1 if dtype == "bf16" else 0, dist, seed, stream, e0, n, T, d,
                                    float(sigma), mask_seed, mask_stream, mask_threshold(mask_p))
        if rc != 0:
            raise ValueError("tda_synth_fill_cpu: bad argument")
        return out
    return _factors_numpy(seed, stream, n, T, d, sigma, dist, e0, dtype, mask_p, mask_seed, mask_stream)


def _factors_numpy(seed, stream, n, T, d, sigma, dist, e0, dtype, mask_p, mask_seed, mask_stream):
    key = stream_key(seed, stream)
    e = np.arange(e0, e0 + n, dtype=np.uint64)[:, None, None]
    t = np.arange(T, dtype=np.uint64)[None, :, None]
    c = np.arange(d, dtype=np.uint64)[None, None, :]
    gen = normal if dist == DIST_NORMAL else student_t4
    v = np.empty((n, T, d), dtype=np.float32)
    flat = v.reshape(-1)
    chunk = max(1, (1 << 16) // max(d, 1))  # token rows per chunk, cache-sized
    rows = (e * np.uint64(T) + t).reshape(-1)  # global token index of each (example, token) row

    def fill(r0):
        r = rows[r0:r0 + chunk, None]
        with np.errstate(over="ignore"):
            idx = r * np.uint64(d) + c.reshape(1, -1)
        flat[r0 * d:(r0 + r.shape[0]) * d] = (gen(key, idx) * np.float32(sigma)).astype(np.float32).reshape(-1)

    starts = range(0, rows.size, chunk)
    if rows.size * d >= (1 << 22):  # numpy releases the GIL: fill chunks on all cores
        from concurrent.futures import ThreadPoolExecutor
        with ThreadPoolExecutor(max_workers=os.cpu_count() or 1) as ex:
            list(ex.map(fill, starts))
    else:
        for r0 in starts:
            fill(r0)
    thr = mask_threshold(mask_p)
    if thr > 0:
        mkey = stream_key(mask_seed, mask_stream)
        with np.errstate(over="ignore"):
            tok = e[:, :, 0] * np.uint64(T) + t[:, :, 0]
        keep = word(mkey, tok) >= np.uint64(thr)
        v = np.where(keep[:, :, None], v, np.float32(0.0)).astype(np.float32)
    if dtype == "bf16":
        return f32_to_bf16_bits(v)
    return v


def to_f64(x: np.ndarray, dtype: str) -> np.ndarray:
    """Widen generator output (fp32, or bf16 bit patterns) to float64, exactly."""
    if dtype == "bf16":
        return bf16_bits_to_f32(x).astype(np.float64)
    return np.asarray(x, dtype=np.float32).astype(np.float64)


# ------------------------------------------------------------------ device side
_synth_lib = None


def _load_device_lib():
    global _synth_lib
    if _synth_lib is None:
        import ctypes
        import os

        path = os.path.join(os.path.dirname(os.path.abspath(__file__)), "libtda_synth.so")
        if not os.path.exists(path):
            raise ImportError(f"{path} is missing: run paper_2609_38767_gb300.build.build() first")
        lib = ctypes.CDLL(path)
        u64, i64, i32 = ctypes.c_uint64, ctypes.c_int64, ctypes.c_int32
        lib.tda_synth_fill.restype = i32
        lib.tda_synth_fill.argtypes = [ctypes.c_void_p, i32, i32, u64, u64, i64, i64, i64, i64,
                                       ctypes.c_float, u64, u64, u64, ctypes.c_void_p]
        _synth_lib = lib
    return _synth_lib


def fill_device(out, seed: int, stream: int, n: int, T: int, d: int, sigma: float = 1.0,
                dist: int = DIST_NORMAL, e0: int = 0, mask_p: float = 0.0,
                mask_seed: int = SEED_MASK, mask_stream: int = 0, cuda_stream=None) -> None:
    """Fill a device tensor (fp32 or bf16, n*T*d elements) with the generator's values."""
    import torch

    dt = {torch.float32: 0, torch.bfloat16: 1}[out.dtype]
    assert out.is_cuda and out.is_contiguous() and out.numel() >= n * T * d
    s = cuda_stream if cuda_stream is not None else torch.cuda.current_stream().cuda_stream
    rc = _load_device_lib().tda_synth_fill(out.data_ptr(), dt, dist, seed, stream, e0, n, T, d,
                                           float(sigma), mask_seed, mask_stream,
                                           mask_threshold(mask_p), s)
    if rc != 0:
        raise RuntimeError(f"tda_synth_fill failed ({rc})")
