"""Quantization and dequantization at a region boundary (Section 3.2,
"partial quantization"): Q nodes map a floating-point tensor T to a
lower-precision tensor T_q with a scale S and a zero point Z, fixed at
compile time from calibration data.

TEST INFRASTRUCTURE.  Plain numpy, written from the definitions of the number
formats; it shares nothing with the CUDA path.

Two target formats:

* 8-bit integers (the fixed-point case the paper's FPGA backends use):
    T_q = clamp(round_half_even(T / S) + Z, -128, 127),   T = (T_q - Z) S.
* FP8 E4M3 (the 8-bit tensor-core format of this GPU; symmetric, Z = 0):
    T_q = e4m3(T * fp32(1 / S)),   T = T_q S,
  where e4m3() rounds to the nearest E4M3 value, ties to even, and clamps to
  the largest finite value 448 (saturating, no infinities).  The product
  T * fp32(1 / S) is formed in fp32, as the accelerator forms it, so that both
  sides take the rounding decision on the same value.

Weights of an FP8 convolution or dense layer are quantized per output
channel k at compile time, after any batch norm is folded into them, with a
power-of-two scale (so that dequantization is exact):
    S_w[k] = 2^ceil(log2(max_c |w'[k, c]| / 448)),   w_q = e4m3(w' / S_w[k]).
"""
from __future__ import annotations

import numpy as np

E4M3_MAX = 448.0           # 1.75 x 2^8
E4M3_MIN_NORMAL = 2.0 ** -6
E4M3_SUBNORMAL_STEP = 2.0 ** -9   # 0.001 x 2^-6


def round_e4m3(x):
    """Nearest FP8 E4M3 value (1 sign bit, 4 exponent bits with bias 7, 3
    mantissa bits), ties to even, saturating at +-448.  From the format: a
    value of magnitude in [2^e, 2^(e+1)) with e >= -6 is a multiple of
    2^(e-3); below 2^-6 the values are the multiples of 2^-9 (subnormals).
    np.rint rounds half to even on the scaled value.  Returns float64."""
    x = np.asarray(x, dtype=np.float64)
    a = np.abs(x)
    _, ex = np.frexp(a)                      # a = m 2^ex, 1/2 <= m < 1: binade 2^(ex-1)
    e = np.maximum(ex.astype(np.int64) - 1, -6)
    step = np.ldexp(1.0, e - 3)
    r = np.rint(a / step) * step
    r = np.minimum(r, E4M3_MAX)
    return np.where(np.isnan(x), np.nan, np.copysign(r, x))


def e4m3_values():
    """Every finite non-negative E4M3 value, ascending (the 127 codes 0x00 ..
    0x7E: subnormals m 2^-9, m = 0..7; normals (1 + m/8) 2^e, e = -6..8,
    except e = 8, m = 7, the NaN code)."""
    vals = [m * 2.0 ** -9 for m in range(8)]
    for e in range(-6, 9):
        for m in range(8):
            if e == 8 and m == 7:
                continue
            vals.append((1 + m / 8.0) * 2.0 ** e)
    return np.array(vals)


def inv_scale_f32(scale: float) -> np.float32:
    """fp32(1 / S): the reciprocal in double, rounded once to fp32."""
    return np.float32(1.0 / np.float64(scale))


def quantize_e4m3(t, scale: float):
    """T_q = e4m3(T * fp32(1/S)) with the product in fp32 (T bf16-exact or fp32)."""
    prod = np.asarray(t, dtype=np.float32) * inv_scale_f32(scale)
    return round_e4m3(prod.astype(np.float64))


def dequantize_e4m3(q, scale: float):
    return np.asarray(q, dtype=np.float64) * np.float64(scale)


def quantize_int8(t, scale: float, zero_point: int):
    q = np.rint(np.asarray(t, dtype=np.float64) / np.float64(scale)) + zero_point
    return np.clip(q, -128, 127)


def dequantize_int8(q, scale: float, zero_point: int):
    return (np.asarray(q, dtype=np.float64) - zero_point) * np.float64(scale)


def weight_scales_e4m3(w_folded):
    """Per-output-channel power-of-two scales: 2^ceil(log2(max|w'[k]| / 448));
    1 for an all-zero channel.  w_folded: [K, ...]."""
    w = np.asarray(w_folded, dtype=np.float64).reshape(len(w_folded), -1)
    m = np.max(np.abs(w), axis=1)
    # smallest power of two S with m / S <= 448: m / 448 = f 2^ex, 1/2 <= f < 1
    f, ex = np.frexp(np.where(m > 0, m / E4M3_MAX, 1.0))
    e = np.where(f == 0.5, ex - 1, ex).astype(np.int64)
    return np.where(m > 0, np.ldexp(1.0, e), 1.0)


def quantize_weights_e4m3(w_folded):
    """(w_q, S_w): w_q = e4m3(w' / S_w[k]) per output channel; dequantized
    weights are w_q S_w[k] exactly."""
    w = np.asarray(w_folded, dtype=np.float64)
    s = weight_scales_e4m3(w)
    shape = (-1,) + (1,) * (w.ndim - 1)
    return round_e4m3(w / s.reshape(shape)), s
