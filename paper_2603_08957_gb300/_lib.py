"""ctypes declarations of the C ABI in include/ucl.h.

Loads the in-tree ``_build/libucl.so`` (building it first if it is missing or
older than its sources).  There is no fallback: if the library cannot be built
or loaded, importing the binding raises.
"""
from __future__ import annotations

import ctypes
import os
import threading

from . import build as _build

UCL_NSTAGES = 4

STATUS_NAMES = {
    0: "UCL_OK",
    1: "UCL_ERR_ARG",
    2: "UCL_ERR_SPEC",
    3: "UCL_ERR_SHAPE",
    4: "UCL_ERR_DUP_KEY",
    5: "UCL_ERR_KEY_RANGE",
    6: "UCL_ERR_OOM",
    7: "UCL_ERR_CUDA",
    8: "UCL_ERR_UNSUPPORTED",
    9: "UCL_ERR_TIMEOUT",
}

# Every symbol include/ucl.h declares.
EXPORTS = [
    "ucl_ctx_create",
    "ucl_ctx_destroy",
    "ucl_ctx_synchronize",
    "ucl_ctx_set_timing",
    "ucl_get_last_stats",
    "ucl_ctx_timings",
    "ucl_ctx_fixup_bytes",
    "ucl_ctx_set_wait_limit",
    "ucl_ctx_withhold_stage",
    "ucl_relation_create",
    "ucl_relation_destroy",
    "ucl_relation_info",
    "ucl_relation_data",
    "ucl_relation_download",
    "ucl_einsum",
    "ucl_repartition",
    "ucl_relation_stats",
    "ucl_drop_zero_tiles",
    "ucl_plan",
    "ucl_plan_dag",
    "ucl_keys_check_noalloc",
    "ucl_status_str",
    "ucl_last_error",
]

ALLOC_FN = ctypes.CFUNCTYPE(ctypes.c_void_p, ctypes.c_size_t, ctypes.c_void_p)
FREE_FN = ctypes.CFUNCTYPE(None, ctypes.c_void_p, ctypes.c_size_t, ctypes.c_void_p)


class EinsumOpts(ctypes.Structure):
    _fields_ = [
        ("out_dtype", ctypes.c_int),
        ("epi", ctypes.c_int),
        ("scale", ctypes.c_float),
        ("path", ctypes.c_int),
        ("agg", ctypes.c_int),
        ("comb", ctypes.c_int),
        ("map", ctypes.c_int),
    ]


class Stats(ctypes.Structure):
    _fields_ = [
        ("n_pairs", ctypes.c_int64),
        ("n_segments", ctypes.c_int64),
        ("flops", ctypes.c_double),
        ("bytes_contract", ctypes.c_double),
        ("path", ctypes.c_int),
        ("launches", ctypes.c_int),
        ("timed", ctypes.c_int),
        ("n_units", ctypes.c_int),
        ("n_bands", ctypes.c_int),
        ("n_band_segments", ctypes.c_int64),
        ("stage_ms", ctypes.c_float * UCL_NSTAGES),
    ]


PLAN_MAX_VERTICES = 64


class PlanVertex(ctypes.Structure):
    _fields_ = [
        ("left", ctypes.c_int),
        ("right", ctypes.c_int),
        ("labels", ctypes.c_char_p),
        ("dtype_bytes", ctypes.c_int),
        ("nnz", ctypes.c_double),
        ("distinct", ctypes.POINTER(ctypes.c_double)),
    ]


class CostModel(ctypes.Structure):
    _fields_ = [
        ("xfer", ctypes.c_double),
        ("flop", ctypes.c_double),
        ("add", ctypes.c_double),
        ("fixed", ctypes.c_double),
        ("key_bytes", ctypes.c_int),
        ("max_call_bytes", ctypes.c_double),
    ]


class PlanChoice(ctypes.Structure):
    _fields_ = [
        ("cost", ctypes.c_double),
        ("up", ctypes.c_uint32 * PLAN_MAX_VERTICES),
        ("in_up", (ctypes.c_uint32 * 2) * PLAN_MAX_VERTICES),
    ]


_lock = threading.Lock()
_lib = None


def _declare(lib):
    c = ctypes
    vp, i64, i32 = c.c_void_p, c.c_int64, c.c_int
    pp = c.POINTER(c.c_void_p)
    lib.ucl_ctx_create.argtypes = [i32, vp, ALLOC_FN, FREE_FN, vp, pp]
    lib.ucl_ctx_destroy.argtypes = [vp]
    lib.ucl_ctx_synchronize.argtypes = [vp]
    lib.ucl_ctx_set_timing.argtypes = [vp, i32]
    lib.ucl_get_last_stats.argtypes = [vp, c.POINTER(Stats)]
    lib.ucl_ctx_timings.argtypes = [vp, c.POINTER(c.c_float), i32, c.POINTER(i32), i32]
    lib.ucl_ctx_fixup_bytes.argtypes = [vp, c.POINTER(i64), i32]
    lib.ucl_ctx_set_wait_limit.argtypes = [vp, i64]
    lib.ucl_ctx_withhold_stage.argtypes = [vp, i32]
    lib.ucl_relation_create.argtypes = [vp, i64, i32, vp, c.POINTER(i64), i32, c.POINTER(i64), i32, vp, i32, pp]
    lib.ucl_relation_destroy.argtypes = [vp]
    lib.ucl_relation_info.argtypes = [vp, c.POINTER(i64), c.POINTER(i32), c.POINTER(i32), c.POINTER(i64),
                                      c.POINTER(i64), c.POINTER(i32)]
    lib.ucl_relation_data.argtypes = [vp, pp, pp]
    lib.ucl_relation_download.argtypes = [vp, vp, vp]
    lib.ucl_einsum.argtypes = [vp, c.c_char_p, i32, pp, c.POINTER(EinsumOpts), pp]
    lib.ucl_repartition.argtypes = [vp, c.c_char_p, vp, pp]
    lib.ucl_relation_stats.argtypes = [vp, vp, c.POINTER(i64), c.POINTER(i64)]
    lib.ucl_drop_zero_tiles.argtypes = [vp, vp, pp]
    lib.ucl_plan.argtypes = [i32, c.POINTER(PlanVertex), c.c_char_p, c.POINTER(i64), i32, c.POINTER(CostModel), i32,
                             c.POINTER(PlanChoice), c.POINTER(i32)]
    lib.ucl_plan_dag.argtypes = [i32, c.POINTER(PlanVertex), c.c_char_p, c.POINTER(i64), i32, c.POINTER(CostModel),
                                 c.POINTER(PlanChoice), c.POINTER(i32)]
    lib.ucl_keys_check_noalloc.argtypes = [i32, vp, i64, i32, vp, c.POINTER(i64), c.POINTER(i32)]
    lib.ucl_status_str.argtypes = [i32]
    lib.ucl_status_str.restype = c.c_char_p
    lib.ucl_last_error.argtypes = [vp]
    lib.ucl_last_error.restype = c.c_char_p
    for name in EXPORTS:
        if name not in ("ucl_status_str", "ucl_last_error"):
            getattr(lib, name).restype = i32


def library_path() -> str:
    return _build.LIB


def load():
    """Build (if stale) and load libucl.so; raises if that is impossible."""
    global _lib
    with _lock:
        if _lib is None:
            path = _build.build()
            if not os.path.exists(path):
                raise ImportError(f"libucl.so not found at {path}")
            lib = ctypes.CDLL(path)
            _declare(lib)
            _lib = lib
    return _lib
