"""GB300-native routine-selecting CNN inference (SoftNeuro, arXiv 2110.06037).

Layers are served by interchangeable routines (hand-written sm_103a kernels);
a profiler measures each routine and DPRS (Alg. 1) picks the fastest routine
path, counting the adapt (cast / layout) conversions between layers.  The
work happens in libsn.so behind the C ABI in include/sn.h; this package is a
thin binding over it.

Schemas are (dtype, layout) pairs: dtype "f32" | "f16" | "bf16" | "qi8"
(symmetric int8 codes with one scale per blob: Graph.set_qscale or
Graph.calibrate), layout "nchw" | "nhwc".  Nets may have several inputs
(Graph.add_input) and outputs (Graph.set_outputs, Graph.run_multi).
"""
from ._sn import (SN_SELECT_BRUTE, SN_SELECT_DPRS, SN_OPT_CHAIN, SN_OPT_CHECK, SN_OPT_CUDA_GRAPH, SN_OPT_WAIT_LIMIT, SN_OPT_SHARE_BUFFERS, SnError, lib,
                  routine_name, variant_name)
from .api import Graph, convert, convert_q, storage_shape
from .netbuild import build_graph, fuse_residual, fused_description

__all__ = ["Graph", "convert", "convert_q", "build_graph", "fuse_residual", "fused_description", "storage_shape", "SnError", "lib", "routine_name",
           "variant_name", "SN_SELECT_DPRS", "SN_SELECT_BRUTE", "SN_OPT_CHAIN", "SN_OPT_CHECK", "SN_OPT_CUDA_GRAPH", "SN_OPT_WAIT_LIMIT", "SN_OPT_SHARE_BUFFERS"]
