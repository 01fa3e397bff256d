"""ctypes binding of libsn.so (include/sn.h), same names as the C ABI.

This module only marshals arguments: every step of profiling, selection and
inference runs inside the library.  If libsn.so has not been built the import
of the library fails loudly; there is no fallback.
"""
from __future__ import annotations

import ctypes as C
import os

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "libsn.so")

SN_OK, SN_EINVAL, SN_ENOMEM, SN_ECUDA, SN_EUNSUPPORTED, SN_ESTATE, SN_ETIMEOUT, SN_EINFEASIBLE = range(8)
STATUS_NAMES = ["SN_OK", "SN_EINVAL", "SN_ENOMEM", "SN_ECUDA", "SN_EUNSUPPORTED", "SN_ESTATE",
                "SN_ETIMEOUT", "SN_EINFEASIBLE"]
SN_F32, SN_F16, SN_BF16, SN_QI8 = 0, 1, 2, 3
SN_NCHW, SN_NHWC = 0, 1
SN_L_CONV2, SN_L_DWCONV2, SN_L_MAXPOOL, SN_L_GAP, SN_L_ADD, SN_L_DENSE, SN_L_MUL = range(7)
SN_ACT = {"none": 0, None: 0, "relu": 1, "relu6": 2, "hswish": 3, "hsigmoid": 4}
SN_SELECT_DPRS, SN_SELECT_BRUTE = 0, 1
SN_OPT_CUDA_GRAPH, SN_OPT_CHECK, SN_OPT_CHAIN, SN_OPT_WAIT_LIMIT, SN_OPT_SHARE_BUFFERS = 0, 1, 2, 3, 4
COST_INF = np.iinfo(np.int64).max

DTYPES = {"f32": SN_F32, "f16": SN_F16, "bf16": SN_BF16, "qi8": SN_QI8}
LAYOUTS = {"nchw": SN_NCHW, "nhwc": SN_NHWC}


class sn_schema(C.Structure):
    _fields_ = [("dtype", C.c_int32), ("layout", C.c_int32)]


class sn_conv_params(C.Structure):
    _fields_ = [(n, C.c_int32) for n in ("c_in", "c_out", "kh", "kw", "sh", "sw", "ph", "pw", "dh", "dw",
                                        "groups", "act")]


class sn_pool_params(C.Structure):
    _fields_ = [(n, C.c_int32) for n in ("kh", "kw", "sh", "sw", "ph", "pw")]


class sn_add_params(C.Structure):
    _fields_ = [("act", C.c_int32)]


class sn_dense_params(C.Structure):
    _fields_ = [("in_features", C.c_int32), ("out_features", C.c_int32), ("act", C.c_int32)]


class sn_candidate(C.Structure):
    _fields_ = [("routine", C.c_int32), ("variant", C.c_int32), ("schema", C.c_int32),
                ("layer", C.c_int32), ("cost_ns", C.c_int64), ("out_schema", C.c_int32)]


class sn_cost_table(C.Structure):
    _fields_ = [("n_layers", C.c_int32), ("n_schemas", C.c_int32), ("n_edges", C.c_int32),
                ("n_candidates", C.c_int32), ("candidates", C.POINTER(sn_candidate)),
                ("edges", C.POINTER(C.c_int32)), ("adapt_cost", C.POINTER(C.c_int64))]


class sn_path(C.Structure):
    _fields_ = [("total_ns", C.c_int64), ("n_layers", C.c_int32),
                ("schema", C.POINTER(C.c_int32)), ("candidate", C.POINTER(C.c_int32))]


class sn_profile_opts(C.Structure):
    _fields_ = [("warmup", C.c_int32), ("iters", C.c_int32), ("topk", C.c_int32), ("passes", C.c_int32)]


ALLOC_FN = C.CFUNCTYPE(C.c_void_p, C.c_size_t, C.c_void_p)
FREE_FN = C.CFUNCTYPE(None, C.c_void_p, C.c_void_p)

# exported symbol -> (restype, argtypes)
SIGNATURES = {
    "sn_graph_create": (C.c_int, [C.POINTER(C.c_int64), sn_schema, sn_schema, C.POINTER(sn_schema), C.c_int32,
                                  ALLOC_FN, FREE_FN, C.c_void_p, C.POINTER(C.c_void_p)]),
    "sn_add_layer": (C.c_int, [C.c_void_p, C.c_int32, C.c_void_p, C.POINTER(C.c_int32), C.c_int32,
                               C.c_void_p, C.c_void_p, C.POINTER(C.c_int32)]),
    "sn_get_cost_table": (C.c_int, [C.c_void_p, C.POINTER(sn_cost_table)]),
    "sn_set_cost_table": (C.c_int, [C.c_void_p, C.POINTER(sn_cost_table)]),
    "sn_get_schema": (C.c_int, [C.c_void_p, C.c_int32, C.POINTER(sn_schema), C.POINTER(C.c_int32)]),
    "sn_profile": (C.c_int, [C.c_void_p, C.POINTER(sn_profile_opts), C.c_void_p]),
    "sn_select_path": (C.c_int, [C.c_void_p, C.c_int32, C.POINTER(sn_path)]),
    "sn_set_path": (C.c_int, [C.c_void_p, C.POINTER(C.c_int32), C.c_int32]),
    "sn_set_option": (C.c_int, [C.c_void_p, C.c_int32, C.c_int64]),
    "sn_run": (C.c_int, [C.c_void_p, C.c_void_p, C.c_void_p, C.c_void_p]),
    "sn_run_host": (C.c_int, [C.c_void_p, C.c_void_p, C.c_void_p, C.c_void_p]),
    "sn_fuse_residual": (C.c_int, [C.c_void_p, C.POINTER(C.c_int32), C.c_int32, C.POINTER(C.c_int32)]),
    "sn_run_timed": (C.c_int, [C.c_void_p, C.c_void_p, C.c_void_p, C.c_void_p, C.POINTER(C.c_float),
                               C.POINTER(C.c_float)]),
    "sn_layer_shape": (C.c_int, [C.c_void_p, C.c_int32, C.POINTER(C.c_int64)]),
    "sn_plan_stats": (C.c_int, [C.c_void_p, C.POINTER(C.c_int32), C.POINTER(C.c_int32), C.c_void_p]),
    "sn_plan_memory": (C.c_int, [C.c_void_p, C.POINTER(C.c_int64), C.POINTER(C.c_int64), C.c_void_p]),
    "sn_save_plan": (C.c_int, [C.c_void_p, C.c_char_p]),
    "sn_load_plan": (C.c_int, [C.c_void_p, C.c_char_p]),
    "sn_graph_destroy": (None, [C.c_void_p]),
    "sn_routine_name": (C.c_char_p, [C.c_int32]),
    "sn_variant_name": (C.c_char_p, [C.c_int32, C.c_int32]),
    "sn_candidate_desc": (C.c_char_p, [C.c_void_p, C.c_int32]),
    "sn_convert": (C.c_int, [C.c_void_p, sn_schema, C.c_void_p, sn_schema, C.POINTER(C.c_int64), C.c_void_p]),
    "sn_convert_q": (C.c_int, [C.c_void_p, sn_schema, C.c_void_p, sn_schema, C.POINTER(C.c_int64), C.c_float,
                               C.c_void_p]),
    "sn_set_qscale": (C.c_int, [C.c_void_p, C.c_int32, C.c_float]),
    "sn_get_qscale": (C.c_int, [C.c_void_p, C.c_int32, C.POINTER(C.c_float)]),
    "sn_calibrate": (C.c_int, [C.c_void_p, C.c_void_p, C.c_void_p]),
    "sn_add_input": (C.c_int, [C.c_void_p, C.POINTER(C.c_int64), C.POINTER(C.c_int32)]),
    "sn_set_outputs": (C.c_int, [C.c_void_p, C.POINTER(C.c_int32), C.c_int32]),
    "sn_get_io": (C.c_int, [C.c_void_p, C.POINTER(C.c_int32), C.POINTER(C.c_int32)]),
    "sn_run_multi": (C.c_int, [C.c_void_p, C.POINTER(C.c_void_p), C.c_int32, C.POINTER(C.c_void_p), C.c_int32,
                               C.c_void_p]),
    "sn_conv2d_wino_noalloc": (C.c_int, [C.c_void_p, sn_schema, C.POINTER(C.c_int64), C.c_int32, C.c_int32,
                                         C.c_int32, C.c_void_p, C.c_void_p, C.c_void_p, C.c_void_p]),
    "sn_last_error": (C.c_char_p, []),
}
NOALLOC_SCRATCH_BYTES = 32 * 1024 * 1024

_lib = None


class SnError(RuntimeError):
    def __init__(self, status, msg):
        super().__init__(f"{STATUS_NAMES[status] if 0 <= status < 8 else status}: {msg}")
        self.status = status


def lib():
    """The loaded libsn.so.  Raises if the library was not built."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise ImportError(f"{LIB_PATH} is missing: build it with paper_2110_06037_gb300.build.build() "
                              "(there is no fallback path)")
        L = C.CDLL(LIB_PATH)
        for name, (res, args) in SIGNATURES.items():
            f = getattr(L, name)
            f.restype = res
            f.argtypes = args
        _lib = L
    return _lib


def check(status):
    if status != SN_OK:
        raise SnError(status, lib().sn_last_error().decode())


def schema(s) -> sn_schema:
    """('f16', 'nhwc') -> sn_schema."""
    if isinstance(s, sn_schema):
        return s
    dt, lay = s
    return sn_schema(DTYPES[dt], LAYOUTS[lay])


def routine_name(r: int) -> str:
    v = lib().sn_routine_name(r)
    return v.decode() if v is not None else "?"


def variant_name(r: int, v: int) -> str:
    s = lib().sn_variant_name(r, v)
    return s.decode() if s is not None else "?"
