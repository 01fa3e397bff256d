"""CPU oracle for the SoftNeuro hot path (arXiv 2110.06037).

TEST INFRASTRUCTURE ONLY: the product library never imports, links or runs
anything in this package.  Only the tests, the smoke check and the benchmark's
CPU-baseline leg use it.  It shares no code with the CUDA path; both sides are
fed the same seeded arrays by the caller.

Numerics are plain fp64 definitions (sn_oracle.c); the path search is the
exhaustive argmin of Def. 2 / Eq. 2 (sn_oracle.c) plus an independent exact
block-wise search for nets too large to enumerate (paths.py).
"""
from __future__ import annotations

import ctypes
import os
import subprocess

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "sn_oracle.c")
_LIB_PATH = os.path.join(_HERE, "liboracle.so")

GCC_CMD = ["gcc", "-O2", "-std=c11", "-fopenmp", "-ffp-contract=off", "-fPIC", "-shared",
           _SRC, "-o", _LIB_PATH, "-lm"]

ACT = {"none": 0, "relu": 1, "relu6": 2, "hswish": 3, "hsigmoid": 4, None: 0}
INF = np.iinfo(np.int64).max

_lib = None


def build(force: bool = False) -> str:
    """Compile sn_oracle.c into liboracle.so next to it (gcc + OpenMP)."""
    if force or not os.path.exists(_LIB_PATH) or \
            os.path.getmtime(_LIB_PATH) < os.path.getmtime(_SRC):
        subprocess.run(GCC_CMD, check=True)
    return _LIB_PATH


def lib():
    global _lib
    if _lib is None:
        build()
        L = ctypes.CDLL(_LIB_PATH)
        i64, i32, dp = ctypes.c_int64, ctypes.c_int32, ctypes.c_void_p
        L.or_conv_out_dim.restype = i64
        L.or_conv_out_dim.argtypes = [i64] * 5
        L.or_conv2d.restype = ctypes.c_int
        L.or_conv2d.argtypes = [dp, i64, i64, i64, i64, dp, dp, i64, i64, i64,
                                i64, i64, i64, i64, i64, i64, i64, ctypes.c_int, dp]
        L.or_maxpool2d.restype = ctypes.c_int
        L.or_maxpool2d.argtypes = [dp, i64, i64, i64, i64, i64, i64, i64, i64, i64, i64, dp]
        L.or_gap.restype = None
        L.or_gap.argtypes = [dp, i64, i64, i64, i64, dp]
        L.or_add.restype = None
        L.or_add.argtypes = [dp, dp, i64, ctypes.c_int, dp]
        L.or_dense.restype = None
        L.or_dense.argtypes = [dp, dp, dp, i64, i64, i64, ctypes.c_int, dp]
        L.or_mul.restype = None
        L.or_mul.argtypes = [dp, dp, i64, i64, i64, ctypes.c_int, dp]
        for name in ("or_cast_f32_to_f16", "or_cast_f32_to_bf16",
                     "or_cast_f16_to_f32", "or_cast_bf16_to_f32"):
            getattr(L, name).restype = None
            getattr(L, name).argtypes = [dp, dp, i64]
        for name in ("or_nchw_to_nhwc", "or_nhwc_to_nchw"):
            getattr(L, name).restype = None
            getattr(L, name).argtypes = [dp, dp, i64, i64, i64, i64, i64]
        L.or_fastest_per_schema.restype = None
        L.or_fastest_per_schema.argtypes = [i32, dp, dp, i32, dp]
        L.or_path_cost.restype = i64
        L.or_path_cost.argtypes = [i32, i32, dp, i32, dp, dp, dp]
        L.or_brute_force.restype = i64
        L.or_brute_force.argtypes = [i32, i32, dp, i32, dp, dp, dp, dp]
        _lib = L
    return _lib


def _p(a: np.ndarray):
    return a.ctypes.data_as(ctypes.c_void_p)


def _f64(a) -> np.ndarray:
    return np.ascontiguousarray(np.asarray(a, dtype=np.float64))


# ----------------------------------------------------------------------------
# numerics (all NCHW, fp64)
# ----------------------------------------------------------------------------

def conv_out_dim(n, k, s, p, d=1) -> int:
    return int(lib().or_conv_out_dim(n, k, s, p, d))


def conv2d(x, w, b=None, stride=(1, 1), pad=(0, 0), dil=(1, 1), groups=1, act="none"):
    """conv2 layer: cross-correlation + bias + activation (sections II, III-B)."""
    x, w = _f64(x), _f64(w)
    N, C, H, W = x.shape
    K, Cg, R, S = w.shape
    if Cg * groups != C:
        raise ValueError("weight shape does not match C/groups")
    P = conv_out_dim(H, R, stride[0], pad[0], dil[0])
    Q = conv_out_dim(W, S, stride[1], pad[1], dil[1])
    y = np.empty((N, K, P, Q), np.float64)
    bb = _f64(b) if b is not None else None
    rc = lib().or_conv2d(_p(x), N, C, H, W, _p(w), _p(bb) if bb is not None else None,
                         K, R, S, stride[0], stride[1], pad[0], pad[1], dil[0], dil[1],
                         groups, ACT[act], _p(y))
    if rc:
        raise ValueError("or_conv2d rejected the sizes")
    return y


def maxpool2d(x, k=(3, 3), stride=(2, 2), pad=(1, 1)):
    x = _f64(x)
    N, C, H, W = x.shape
    P = conv_out_dim(H, k[0], stride[0], pad[0])
    Q = conv_out_dim(W, k[1], stride[1], pad[1])
    y = np.empty((N, C, P, Q), np.float64)
    lib().or_maxpool2d(_p(x), N, C, H, W, k[0], k[1], stride[0], stride[1], pad[0], pad[1], _p(y))
    return y


def gap(x):
    x = _f64(x)
    N, C, H, W = x.shape
    y = np.empty((N, C, 1, 1), np.float64)
    lib().or_gap(_p(x), N, C, H, W, _p(y))
    return y


def add(a, b, act="none"):
    a, b = _f64(a), _f64(b)
    if a.shape != b.shape:
        raise ValueError("add operands differ in shape")
    y = np.empty_like(a)
    lib().or_add(_p(a), _p(b), a.size, ACT[act], _p(y))
    return y


def mul(x, s, act="none"):
    """y[n,c,h,w] = act(x[n,c,h,w] * s[n,c]): the scale of a squeeze-and-excite
    block (MobileNetV3); s is [N, C] or [N, C, 1, 1]."""
    x, s = _f64(x), _f64(s)
    N, C, H, W = x.shape
    if s.size != N * C:
        raise ValueError("mul: the scale must hold one value per (image, channel)")
    y = np.empty_like(x)
    lib().or_mul(_p(x), _p(np.ascontiguousarray(s.reshape(N, C))), N, C, H * W, ACT[act], _p(y))
    return y


def dense(x, w, b=None, act="none"):
    """y = act(W x + b), W [out, in]; x is [N, in] or [N, in, 1, 1]."""
    x, w = _f64(x), _f64(w)
    N = x.shape[0]
    xin = x.reshape(N, -1)
    out, fin = w.shape
    if xin.shape[1] != fin:
        raise ValueError("dense input size mismatch")
    y = np.empty((N, out), np.float64)
    bb = _f64(b) if b is not None else None
    lib().or_dense(_p(xin), _p(w), _p(bb) if bb is not None else None, N, fin, out,
                   ACT[act], _p(y))
    return y.reshape(N, out, 1, 1)


# ----------------------------------------------------------------------------
# casts (IEEE-754 round to nearest even) and layouts
# ----------------------------------------------------------------------------

def f32_to_f16_bits(x) -> np.ndarray:
    x = np.ascontiguousarray(np.asarray(x, dtype=np.float32))
    y = np.empty(x.shape, np.uint16)
    lib().or_cast_f32_to_f16(_p(x), _p(y), x.size)
    return y


def f32_to_bf16_bits(x) -> np.ndarray:
    x = np.ascontiguousarray(np.asarray(x, dtype=np.float32))
    y = np.empty(x.shape, np.uint16)
    lib().or_cast_f32_to_bf16(_p(x), _p(y), x.size)
    return y


def f16_bits_to_f32(h) -> np.ndarray:
    h = np.ascontiguousarray(np.asarray(h, dtype=np.uint16))
    y = np.empty(h.shape, np.float32)
    lib().or_cast_f16_to_f32(_p(h), _p(y), h.size)
    return y


def bf16_bits_to_f32(h) -> np.ndarray:
    h = np.ascontiguousarray(np.asarray(h, dtype=np.uint16))
    y = np.empty(h.shape, np.float32)
    lib().or_cast_bf16_to_f32(_p(h), _p(y), h.size)
    return y


def to_bits(x, dtype: str) -> np.ndarray:
    """fp32 values -> stored representation of `dtype` ('f32' returns fp32 itself)."""
    if dtype == "f32":
        return np.ascontiguousarray(np.asarray(x, dtype=np.float32))
    if dtype == "f16":
        return f32_to_f16_bits(x)
    if dtype == "bf16":
        return f32_to_bf16_bits(x)
    raise ValueError(dtype)


def from_bits(h, dtype: str) -> np.ndarray:
    """Stored representation of `dtype` -> exact fp32 values."""
    if dtype == "f32":
        return np.asarray(h, dtype=np.float32)
    if dtype == "f16":
        return f16_bits_to_f32(h)
    if dtype == "bf16":
        return bf16_bits_to_f32(h)
    raise ValueError(dtype)


def round_to(x, dtype: str) -> np.ndarray:
    """Values of x (fp32) as they would be stored in `dtype`, widened exactly."""
    return from_bits(to_bits(x, dtype), dtype)


def nchw_to_nhwc(x) -> np.ndarray:
    x = np.ascontiguousarray(x)
    N, C, H, W = x.shape
    y = np.empty((N, H, W, C), x.dtype)
    lib().or_nchw_to_nhwc(_p(x), _p(y), N, C, H, W, x.itemsize)
    return y


def nhwc_to_nchw(x) -> np.ndarray:
    x = np.ascontiguousarray(x)
    N, H, W, C = x.shape
    y = np.empty((N, C, H, W), x.dtype)
    lib().or_nhwc_to_nchw(_p(x), _p(y), N, C, H, W, x.itemsize)
    return y


# ----------------------------------------------------------------------------
# path search (Eq. 1, Def. 1-2)
# ----------------------------------------------------------------------------

def fastest_per_schema(cand_schema, cand_cost, n_schemas) -> np.ndarray:
    """F_i(lambda) for one layer (Eq. 1)."""
    s = np.ascontiguousarray(np.asarray(cand_schema, dtype=np.int32))
    c = np.ascontiguousarray(np.asarray(cand_cost, dtype=np.int64))
    out = np.empty(n_schemas, np.int64)
    lib().or_fastest_per_schema(len(s), _p(s), _p(c), n_schemas, _p(out))
    return out


def path_cost(layer_cost, edges, adapt_cost, assign) -> int:
    """T(S) of a schema assignment (Def. 1, Eq. 2)."""
    lc = np.ascontiguousarray(layer_cost, dtype=np.int64)
    n, ns = lc.shape
    e = np.ascontiguousarray(np.asarray(edges, dtype=np.int32).reshape(-1, 2))
    ac = np.ascontiguousarray(np.asarray(adapt_cost, dtype=np.int64).reshape(len(e), ns, ns))
    a = np.ascontiguousarray(np.asarray(assign, dtype=np.int32))
    return int(lib().or_path_cost(n, ns, _p(lc), len(e), _p(e), _p(ac), _p(a)))


def brute_force(layer_cost, edges, adapt_cost):
    """Exhaustive S* (Def. 2): returns (cost, assignment, number of minimisers)."""
    lc = np.ascontiguousarray(layer_cost, dtype=np.int64)
    n, ns = lc.shape
    e = np.ascontiguousarray(np.asarray(edges, dtype=np.int32).reshape(-1, 2))
    ac = np.ascontiguousarray(np.asarray(adapt_cost, dtype=np.int64).reshape(len(e), ns, ns))
    best = np.zeros(n, np.int32)
    nmin = ctypes.c_int64(0)
    t = lib().or_brute_force(n, ns, _p(lc), len(e), _p(e), _p(ac), _p(best),
                             ctypes.byref(nmin))
    return int(t), best, int(nmin.value)
