"""ctypes binding of the C ABI in include/byoc.h and include/byoc_plan.h.

Argument marshalling only: every computation happens inside libbyoc.so.  If
the library cannot be built or loaded, ``lib()`` raises -- there is no other
implementation to fall back to.
"""
from __future__ import annotations

import ctypes
import os
import threading
from ctypes import POINTER, c_char_p, c_double, c_float, c_int32, c_int64, c_size_t, c_uint32, c_void_p

ABI_VERSION = 2

# byoc_region_desc.options
OPT_FUSE_DW_PW = 0x1
OPT_REGION_KERNEL = 0x2
OPT_MULTICAST = 0x4
OPT_CLUSTER_SPLIT_K = 0x8

# byoc_status
OK, ERR_INVALID_ARG, ERR_UNSUPPORTED, ERR_CUDA, ERR_OOM, ERR_TIMEOUT = range(6)
STATUS_NAMES = {0: "OK", 1: "INVALID_ARG", 2: "UNSUPPORTED", 3: "CUDA", 4: "OOM", 5: "TIMEOUT"}

BF16, FP32, E4M3 = 0, 1, 2
LAYOUT_NHWC, LAYOUT_NC = 0, 1

OP_CONV2D, OP_DENSE, OP_BIAS_ADD, OP_BATCH_NORM, OP_RELU, OP_RELU6, OP_GELU, OP_ADD, OP_QUANTIZE = range(9)

LAUNCH_GEMM, LAUNCH_DEPTHWISE, LAUNCH_S2D, LAUNCH_DWPW, LAUNCH_CHAIN, LAUNCH_QUANT = range(6)
PLAN_MAX_LAUNCHES = 128


class ByocError(RuntimeError):
    def __init__(self, status: int, message: str):
        super().__init__(f"{STATUS_NAMES.get(status, status)}: {message}")
        self.status = status


class Tensor(ctypes.Structure):
    _fields_ = [("ndim", c_int32), ("shape", c_int64 * 4), ("dtype", c_int32), ("layout", c_int32)]


class Op(ctypes.Structure):
    _fields_ = [("kind", c_int32), ("n_in", c_int32), ("in_", c_int32 * 3), ("out", c_int32),
                ("kernel", c_int32 * 2), ("stride", c_int32 * 2), ("pad", c_int32 * 4),
                ("dilation", c_int32 * 2), ("groups", c_int32), ("eps", c_float),
                ("consts", c_void_p * 4)]


class RegionDesc(ctypes.Structure):
    _fields_ = [("abi_version", c_uint32), ("name", c_char_p), ("n_tensors", c_int32),
                ("tensors", POINTER(Tensor)), ("n_ops", c_int32), ("ops", POINTER(Op)),
                ("n_inputs", c_int32), ("input_ids", POINTER(c_int32)), ("n_outputs", c_int32),
                ("output_ids", POINTER(c_int32)), ("options", c_uint32)]


class Info(ctypes.Structure):
    _fields_ = [("flops", c_double), ("bytes", c_double), ("workspace_bytes", c_size_t),
                ("const_bytes", c_size_t), ("n_launches", c_int32), ("n_inputs", c_int32),
                ("n_outputs", c_int32)]


_L = PLAN_MAX_LAUNCHES


class PlanReport(ctypes.Structure):
    _fields_ = [("n_launches", c_int32), ("kind", c_int32 * _L), ("first_op", c_int32 * _L),
                ("n_ops", c_int32 * _L), ("act", c_int32 * _L), ("residual", c_int32 * _L),
                ("gemm_m", c_int32 * _L), ("gemm_n", c_int32 * _L), ("gemm_k", c_int32 * _L),
                ("tile_n", c_int32 * _L), ("tile_k", c_int32 * _L), ("im2col", c_int32 * _L),
                ("grid", c_int32 * _L), ("resident_b", c_int32 * _L), ("slab_slots", c_int32 * _L),
                ("splits", c_int32 * _L), ("pair_units", c_int32 * _L), ("stages", c_int32 * _L),
                ("units", c_int32 * _L), ("fp8", c_int32 * _L), ("multicast", c_int32 * _L),
                ("flops", c_double), ("bytes", c_double),
                ("const_bytes", c_size_t), ("workspace_bytes", c_size_t)]


# Every function the headers declare: name -> (restype, argtypes)
_SIGNATURES = {
    "byoc_compile": (c_int32, [POINTER(RegionDesc), POINTER(c_void_p)]),
    "byoc_run": (c_int32, [c_void_p, POINTER(c_void_p), POINTER(c_void_p), c_void_p]),
    "byoc_check": (c_int32, [c_void_p]),
    "byoc_release": (None, [c_void_p]),
    "byoc_last_error": (c_char_p, []),
    "byoc_query": (c_int32, [c_void_p, POINTER(Info)]),
    "byoc_max_pool2d_nhwc": (c_int32, [c_void_p, c_void_p] + [c_int32] * 7 + [c_void_p]),
    "byoc_global_avg_pool_nhwc": (c_int32, [c_void_p, c_void_p] + [c_int32] * 4 + [c_void_p]),
    "byoc_device_info": (c_int32, [POINTER(c_int32), POINTER(c_int32), POINTER(c_int32)]),
    "byoc_trace_begin": (c_int32, [c_void_p, c_int32]),
    "byoc_trace_end": (c_int32, []),
    "byoc_ffn_noalloc": (c_int32, [c_void_p, c_int32, c_int32, c_int32, c_void_p, c_void_p,
                                   c_void_p, c_void_p, c_void_p, c_void_p]),
    "byoc_plan": (c_int32, [POINTER(RegionDesc), c_int32, POINTER(PlanReport)]),
    "byoc_plan_constants": (c_int32, [POINTER(RegionDesc), c_int32, c_int32, c_int32, c_void_p,
                                      c_size_t, POINTER(c_size_t)]),
    "byoc_nchw_to_nhwc_bf16": (c_int32, [c_void_p, c_void_p] + [c_int32] * 5 + [c_void_p]),
    "byoc_serialize": (c_int32, [c_void_p, c_void_p, c_size_t, POINTER(c_size_t)]),
    "byoc_deserialize": (c_int32, [c_void_p, c_size_t, POINTER(c_void_p)]),
    "byoc_plan_serialize": (c_int32, [POINTER(RegionDesc), c_int32, c_void_p, c_size_t,
                                      POINTER(c_size_t)]),
    "byoc_plan_deserialize": (c_int32, [c_void_p, c_size_t, POINTER(PlanReport)]),
}

_lib = None
_lock = threading.Lock()


def lib_path() -> str:
    return os.path.join(os.path.dirname(os.path.abspath(__file__)), "libbyoc.so")


def lib(build_if_missing: bool = True):
    """Load libbyoc.so (compiling it in-tree first if it is absent)."""
    global _lib
    with _lock:
        if _lib is None:
            path = lib_path()
            if build_if_missing:
                from . import build as _build
                path = _build.build()
            if not os.path.exists(path):
                raise ByocError(ERR_CUDA, f"libbyoc.so not found at {path}; run the build")
            L = ctypes.CDLL(path)
            for name, (res, args) in _SIGNATURES.items():
                f = getattr(L, name)
                f.restype = res
                f.argtypes = args
            _lib = L
    return _lib


def check(status: int) -> None:
    if status != OK:
        msg = lib().byoc_last_error()
        raise ByocError(status, msg.decode() if msg else "")


def declared_symbols():
    return sorted(_SIGNATURES)


def device_info():
    sms, ma, mi = c_int32(), c_int32(), c_int32()
    check(lib().byoc_device_info(ctypes.byref(sms), ctypes.byref(ma), ctypes.byref(mi)))
    return sms.value, ma.value, mi.value


def _stream_ptr(stream) -> int:
    if stream is None:
        import torch
        return torch.cuda.current_stream().cuda_stream
    if isinstance(stream, int):
        return stream
    return stream.cuda_stream


def max_pool2d_nhwc(x, y, k: int, s: int, p: int, stream=None) -> None:
    N, H, W, C = x.shape
    check(lib().byoc_max_pool2d_nhwc(x.data_ptr(), y.data_ptr(), N, H, W, C, k, s, p,
                                     _stream_ptr(stream)))


def global_avg_pool_nhwc(x, y, stream=None) -> None:
    N, H, W, C = x.shape
    check(lib().byoc_global_avg_pool_nhwc(x.data_ptr(), y.data_ptr(), N, H, W, C,
                                          _stream_ptr(stream)))
