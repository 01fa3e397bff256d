"""GB300-native routine-selecting CNN inference (SoftNeuro, arXiv 2110.06037).

Layers are served by interchangeable routines (hand-written sm_103a kernels);
a profiler measures each routine and DPRS (Alg. 1) picks the fastest routine
path, counting the adapt (cast / layout) conversions between layers.  The
work happens in libsn.so behind the C ABI in include/sn.h; this package is a
thin binding over it.
"""
from ._sn import (SN_SELECT_BRUTE, SN_SELECT_DPRS, SN_OPT_CHECK, SN_OPT_CUDA_GRAPH, SnError, lib,
                  routine_name, variant_name)
from .api import Graph, convert, convert_q, storage_shape
from .netbuild import build_graph, fuse_residual

__all__ = ["Graph", "convert", "convert_q", "build_graph", "fuse_residual", "storage_shape", "SnError", "lib", "routine_name",
           "variant_name", "SN_SELECT_DPRS", "SN_SELECT_BRUTE", "SN_OPT_CHECK", "SN_OPT_CUDA_GRAPH"]
