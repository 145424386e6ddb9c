"""ctypes wrappers of the fp64 direct-loop operators in ``byoc_oracle.c``.

TEST INFRASTRUCTURE (see the package docstring).  Every wrapper takes and
returns float64 numpy arrays; shapes follow NHWC / OIHW / [units, in].
"""
from __future__ import annotations

import ctypes
from typing import Sequence

import numpy as np

from . import build as _build

_lib = None

_D = ctypes.POINTER(ctypes.c_double)
_I = ctypes.c_int
_L = ctypes.c_long


def lib():
    global _lib
    if _lib is None:
        _lib = ctypes.CDLL(_build.build())
        _lib.oracle_num_threads.restype = ctypes.c_int
    return _lib


def _p(a: np.ndarray):
    return a.ctypes.data_as(_D)


def _f64(a) -> np.ndarray:
    return np.ascontiguousarray(a, dtype=np.float64)


def num_threads() -> int:
    return int(lib().oracle_num_threads())


def set_num_threads(n: int) -> None:
    lib().oracle_set_num_threads(_I(int(n)))


def conv_out_hw(H, W, R, S, strides, padding, dilation):
    sh, sw = strides
    pt, pl, pb, pr = padding
    dh, dw = dilation
    Ho = (H + pt + pb - dh * (R - 1) - 1) // sh + 1
    Wo = (W + pl + pr - dw * (S - 1) - 1) // sw + 1
    return Ho, Wo


def conv2d_nhwc(x, w, strides=(1, 1), padding=(0, 0, 0, 0), dilation=(1, 1), groups=1):
    """Cross-correlation conv2d; x NHWC, w OIHW (I = C / groups)."""
    x = _f64(x)
    w = _f64(w)
    N, H, W, C = x.shape
    K, Cg, R, S = w.shape
    assert Cg * groups == C and K % groups == 0
    Ho, Wo = conv_out_hw(H, W, R, S, strides, padding, dilation)
    y = np.empty((N, Ho, Wo, K), dtype=np.float64)
    lib().oracle_conv2d_nhwc(_p(x), _I(N), _I(H), _I(W), _I(C), _p(w), _I(K), _I(R), _I(S),
                             _I(groups), _I(strides[0]), _I(strides[1]), _I(padding[0]),
                             _I(padding[1]), _I(padding[2]), _I(padding[3]), _I(dilation[0]),
                             _I(dilation[1]), _p(y))
    return y


def conv2d_nhwc_sampled(x, w, pix: Sequence[int], ks: Sequence[int], strides=(1, 1),
                        padding=(0, 0, 0, 0), dilation=(1, 1), groups=1):
    """conv2d evaluated only at (flattened output pixel, output channel) pairs."""
    x = _f64(x)
    w = _f64(w)
    N, H, W, C = x.shape
    K, Cg, R, S = w.shape
    pix = np.ascontiguousarray(pix, dtype=np.int64)
    ks = np.ascontiguousarray(ks, dtype=np.int32)
    out = np.empty(len(pix), dtype=np.float64)
    lib().oracle_conv2d_nhwc_sampled(
        _p(x), _I(N), _I(H), _I(W), _I(C), _p(w), _I(K), _I(R), _I(S), _I(groups),
        _I(strides[0]), _I(strides[1]), _I(padding[0]), _I(padding[1]), _I(padding[2]),
        _I(padding[3]), _I(dilation[0]), _I(dilation[1]),
        pix.ctypes.data_as(ctypes.POINTER(ctypes.c_long)),
        ks.ctypes.data_as(ctypes.POINTER(ctypes.c_int)), _L(len(pix)), _p(out))
    return out


def dense(x, w):
    """y = x . w^T with w [units, in]."""
    x = _f64(x)
    w = _f64(w)
    M, I = x.shape
    U, I2 = w.shape
    assert I == I2
    y = np.empty((M, U), dtype=np.float64)
    lib().oracle_dense(_p(x), _I(M), _I(I), _p(w), _I(U), _p(y))
    return y


def bias_add(y, b):
    y = _f64(y).copy()
    C = y.shape[-1]
    lib().oracle_bias_add(_p(y), _L(y.size // C), _I(C), _p(_f64(b)))
    return y


def batch_norm(y, gamma, beta, mean, var, eps=1e-5):
    y = _f64(y).copy()
    C = y.shape[-1]
    lib().oracle_batch_norm(_p(y), _L(y.size // C), _I(C), _p(_f64(gamma)), _p(_f64(beta)),
                            _p(_f64(mean)), _p(_f64(var)), ctypes.c_double(eps))
    return y


def relu(y):
    y = _f64(y).copy()
    lib().oracle_relu(_p(y), _L(y.size))
    return y


def relu6(y):
    y = _f64(y).copy()
    lib().oracle_relu6(_p(y), _L(y.size))
    return y


def gelu(y):
    y = _f64(y).copy()
    lib().oracle_gelu(_p(y), _L(y.size))
    return y


def add(a, b):
    y = _f64(a).copy()
    b = _f64(b)
    assert y.shape == b.shape
    lib().oracle_add(_p(y), _p(b), _L(y.size))
    return y


def max_pool2d_nhwc(x, pool_size, strides, padding):
    x = _f64(x)
    N, H, W, C = x.shape
    R, S = pool_size
    Ho = (H + padding[0] + padding[2] - R) // strides[0] + 1
    Wo = (W + padding[1] + padding[3] - S) // strides[1] + 1
    y = np.empty((N, Ho, Wo, C), dtype=np.float64)
    lib().oracle_max_pool2d_nhwc(_p(x), _I(N), _I(H), _I(W), _I(C), _I(R), _I(S),
                                 _I(strides[0]), _I(strides[1]), _I(padding[0]), _I(padding[1]),
                                 _I(padding[2]), _I(padding[3]), _p(y))
    return y


def global_avg_pool_nhwc(x):
    x = _f64(x)
    N, H, W, C = x.shape
    y = np.empty((N, C), dtype=np.float64)
    lib().oracle_global_avg_pool_nhwc(_p(x), _I(N), _I(H), _I(W), _I(C), _p(y))
    return y


def round_bf16(x):
    """Round to the nearest bfloat16 value, ties to even (8 significant bits,
    fp32's exponent range): the cast at a region boundary (Section 3.2,
    "partial quantization" read as fp32 -> bf16).  Written from the
    definition: x = m 2^e with 1/2 <= |m| < 1, so the bf16 neighbours of x are
    the multiples of 2^(e-8) and np.rint picks the nearest, ties to the even
    multiple.  Below 2^-126 the spacing stays 2^-133 (subnormals); beyond the
    largest finite bf16 the result is infinite.  Returns float64."""
    x = _f64(x)
    m, e = np.frexp(x)
    e = np.maximum(e, -125)                      # subnormal range: fixed spacing 2^-133
    q = np.rint(np.ldexp(x, 8 - e))
    r = np.ldexp(q, e - 8)
    bf16_max = (2.0 - 2.0 ** -7) * 2.0 ** 127
    r = np.where(np.abs(r) > bf16_max, np.copysign(np.inf, x), r)
    return np.where(np.isfinite(x), r, x)


def nchw_to_nhwc(x, c_pad):
    """Layout transformation at a region boundary (Section 3.2): NCHW ->
    NHWC with channels zero-padded to c_pad, values rounded to bf16."""
    x = _f64(x)
    N, C, H, W = x.shape
    y = np.zeros((N, H, W, c_pad))
    y[..., :C] = np.transpose(x, (0, 2, 3, 1))
    return round_bf16(y)
