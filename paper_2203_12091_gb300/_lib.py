"""ctypes view of libfxpq.so (include/fxpq.h).  Argument marshalling only.

Loading fails loudly: there is no CPU fallback.  If the library has not been built, call
``paper_2203_12091_gb300.build.build()`` (``__graft_entry__.build()`` does) first.
"""
from __future__ import annotations

import ctypes
import os

from .build import LIB

I32, I64, SZ, VP = ctypes.c_int32, ctypes.c_int64, ctypes.c_size_t, ctypes.c_void_p


class Fmt(ctypes.Structure):
    _fields_ = [("bits", I32), ("is_signed", I32), ("fl", I32)]

    def tup(self):
        return (self.bits, self.is_signed, self.fl)

    def __repr__(self):
        return f"Fmt(bits={self.bits}, S={self.is_signed}, fl={self.fl})"


class Stats(ctypes.Structure):
    _fields_ = [("min", ctypes.c_float), ("max", ctypes.c_float), ("is_signed", I32), ("nonfinite", I32),
                ("sum", ctypes.c_double), ("sumsq", ctypes.c_double), ("n", I64)]


class FlSearchItem(ctypes.Structure):
    _fields_ = [("d_x", VP), ("n", I64), ("is_signed", I32), ("k_lo", I32), ("k_hi", I32), ("fl_lo", I32),
                ("fl_hi", I32), ("d_err", VP), ("d_best", VP), ("d_stats", VP), ("score", I32)]


class QuantizeItem(ctypes.Structure):
    _fields_ = [("d_x", VP), ("d_out", VP), ("kind", I32), ("bits", I32), ("rows", I64), ("C", I32), ("Cp", I32),
                ("rows_per_group", I32), ("reserved", I32), ("d_fl", VP), ("d_stats", VP), ("d_l1", VP)]


class ConvDesc(ctypes.Structure):
    _fields_ = [("N", I32), ("H", I32), ("W", I32), ("C", I32), ("Cp", I32), ("K", I32), ("R", I32), ("S", I32),
                ("stride", I32), ("pad", I32), ("relu", I32), ("out_mode", I32),
                ("fmt_x", Fmt), ("fmt_w", Fmt), ("fmt_b", Fmt), ("fmt_y", Fmt), ("w_l1", I64),
                ("fmt_scale", Fmt), ("fmt_shift", Fmt), ("d_scale", VP), ("d_shift", VP), ("d_wpacked", VP)]


class OpDesc(ctypes.Structure):
    _fields_ = [("op", I32), ("src0", I32), ("src1", I32), ("dst", I32), ("K", I32), ("R", I32), ("S", I32),
                ("stride", I32), ("pad", I32), ("relu", I32), ("last", I32), ("recip_code", I32),
                ("fmt_w", Fmt), ("fmt_b", Fmt), ("fmt_y", Fmt), ("d_w", VP), ("d_bias", VP), ("w_l1", I64),
                ("fmt_scale", Fmt), ("fmt_shift", Fmt), ("d_scale", VP), ("d_shift", VP), ("d_wpacked", VP)]


class DsItem(ctypes.Structure):
    _fields_ = [("d_x", VP), ("d_out", VP), ("nu", I64), ("n_samples", I32), ("fmt", Fmt)]


class CostTerm(ctypes.Structure):
    _fields_ = [("offset", I64), ("nu", I64), ("n_samples", I32), ("layer", I32)]


class ConvF32Desc(ctypes.Structure):
    _fields_ = [("N", I32), ("H", I32), ("W", I32), ("C", I32), ("K", I32), ("R", I32), ("S", I32),
                ("stride", I32), ("pad", I32), ("relu", I32)]


class Net(ctypes.Structure):
    _fields_ = [("n_ops", I32), ("n_slots", I32), ("C", I32), ("H", I32), ("W", I32), ("Cp_in", I32),
                ("fmt_in", Fmt), ("ops", ctypes.POINTER(OpDesc))]


# status / dtype / mode constants (mirror of include/fxpq.h)
OK, ERR_INVALID_ARG, ERR_UNSUPPORTED, ERR_NONFINITE, ERR_TIMEOUT, ERR_CUDA, ERR_WORKSPACE, ERR_RANGE = range(8)
DT_I8, DT_U8, DT_I16, DT_U16, DT_I32, DT_F16 = range(6)
SCORE_L2, SCORE_L1 = 0, 1
OUT_CODES, OUT_ACC64, OUT_F32 = range(3)
QB_ROWS_F16, QB_FLAT_I32 = range(2)
OP_CONV, OP_MAXPOOL, OP_ELTWISE, OP_AVGPOOL = range(4)

_SIGS = {
    "fxpq_quantize": (I32, [VP, I64, Fmt, I32, VP, VP]),
    "fxpq_quantize_rows": (I32, [VP, I64, I32, Fmt, I32, VP, VP]),
    "fxpq_code_l1max": (I32, [VP, I64, I64, VP, VP]),
    "fxpq_fl_search_batch_workspace": (SZ, [I32]),
    "fxpq_fl_search_batch": (I32, [VP, I32, VP, SZ, VP]),
    "fxpq_quantize_batch": (I32, [VP, I32, VP]),
    "fxpq_net_calibrate_workspace": (SZ, [VP, I32]),
    "fxpq_net_calibrate": (I32, [VP, VP, I32, I32, I32, VP, VP, VP, SZ, VP]),
    "fxpq_quantize_images": (I32, [VP, I32, I32, I32, I32, Fmt, I32, VP, VP]),
    "fxpq_fl_search_workspace": (SZ, [I64]),
    "fxpq_fl_search": (I32, [VP, I64, I32, I32, I32, I32, I32, VP, VP, VP, VP, SZ, VP]),
    "fxpq_fl_search_noalloc": (I32, [VP, I64, I32, I32, I32, I32, I32, VP, VP, VP, VP]),
    "fxpq_bn_to_scale": (I32, [VP, VP, VP, VP, I64, ctypes.c_float, VP, VP, VP]),
    "fxpq_pack_codes": (I32, [VP, I64, Fmt, VP, VP]),
    "fxpq_unpack_codes": (I32, [VP, I64, Fmt, VP, VP]),
    "fxpq_packed_weights_bytes": (ctypes.c_size_t, [Fmt, I32, I32]),
    "fxpq_pack_weights": (I32, [VP, Fmt, I32, I32, VP, VP]),
    "fxpq_net_memory": (I32, [ctypes.POINTER(Net), I32, ctypes.POINTER(ctypes.c_double), ctypes.POINTER(ctypes.c_double)]),
    "fxpq_conv_f32": (I32, [ctypes.POINTER(ConvF32Desc), VP, VP, VP, VP, VP]),
    "fxpq_maxpool_f32": (I32, [VP, I32, I32, I32, I32, I32, I32, I32, VP, VP]),
    "fxpq_eltwise_f32": (I32, [VP, VP, I64, I32, VP, VP]),
    "fxpq_avgpool_f32": (I32, [VP, I32, I32, I32, I32, VP, VP]),
    "fxpq_dequantize": (I32, [VP, I64, I32, I32, Fmt, VP, VP]),
    "fxpq_bias_relu_f32": (I32, [VP, I64, I32, VP, I32, VP]),
    "fxpq_ds_stats_batch_workspace": (SZ, [VP, I32]),
    "fxpq_ds_stats_batch": (I32, [VP, I32, VP, SZ, VP]),
    "fxpq_fopt_cost": (I32, [VP, I64, VP, I32, VP, I32, I32, I32, VP, VP]),
    "fxpq_selftest_wait_timeout": (I32, [I64, VP]),
    "fxpq_top1_ties": (I32, [VP, I32, I32, I32, VP, VP]),
    "fxpq_nchw_to_nhwc_f32": (I32, [VP, I32, I32, I32, I32, VP, VP]),
    "fxpq_fl_init": (I32, [ctypes.POINTER(Stats), I32, I32, ctypes.POINTER(Fmt)]),
    "fxpq_conv_workspace": (SZ, [ctypes.POINTER(ConvDesc)]),
    "fxpq_conv_fwd": (I32, [ctypes.POINTER(ConvDesc), VP, VP, VP, VP, ctypes.POINTER(I32), VP, SZ, VP]),
    "fxpq_gemm": (I32, [VP, Fmt, VP, Fmt, VP, Fmt, I32, I32, I32, I32, I32, Fmt, VP, ctypes.POINTER(I32), VP, SZ, VP]),
    "fxpq_maxpool": (I32, [VP, I32, I32, I32, I32, Fmt, I32, I32, I32, VP, VP]),
    "fxpq_eltwise": (I32, [VP, Fmt, VP, Fmt, I64, I32, I32, I32, Fmt, VP, ctypes.POINTER(I32), VP]),
    "fxpq_avgpool": (I32, [VP, I32, I32, I32, I32, Fmt, I32, Fmt, I32, Fmt, VP, ctypes.POINTER(I32), VP]),
    "fxpq_qlayer": (I32, [VP, I64, I32, I32, Fmt, VP, VP]),
    "fxpq_net_workspace": (SZ, [ctypes.POINTER(Net), I32]),
    "fxpq_net_forward": (I32, [ctypes.POINTER(Net), VP, I32, VP, ctypes.POINTER(I32), VP, SZ, VP]),
    "fxpq_get_device_status": (I32, [VP]),
    "fxpq_status_string": (ctypes.c_char_p, [I32]),
    "fxpq_launch_count": (I64, []),
}

_lib = None


def lib():
    """The loaded libfxpq.so.  Raises if it is missing -- there is no fallback path."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB):
            raise RuntimeError(f"libfxpq.so not built ({LIB}); run paper_2203_12091_gb300.build.build()")
        L = ctypes.CDLL(LIB)
        for name, (res, args) in _SIGS.items():
            fn = getattr(L, name)
            fn.restype = res
            fn.argtypes = args
        _lib = L
    return _lib


def declared_symbols():
    return list(_SIGS)


class FxpqError(RuntimeError):
    def __init__(self, where, code):
        msg = lib().fxpq_status_string(code).decode() if _lib is not None else str(code)
        super().__init__(f"{where}: status {code} ({msg})")
        self.code = code


def check(where, code):
    if code != OK:
        raise FxpqError(where, code)
    return code
