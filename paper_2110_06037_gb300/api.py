"""Python front end over the C ABI: Graph (build / profile / select / run).

PyTorch provides device memory (the library's allocator hooks are wired to
the caching allocator) and streams; all computation happens in libsn.so.
Tensors are passed in their schema's storage order: NCHW tensors as
[N, C, H, W], NHWC tensors as [N, H, W, C], contiguous.
"""
from __future__ import annotations

import ctypes as C

import numpy as np

from . import _sn
from ._sn import check, lib

TORCH_DTYPES = {"f32": "float32", "f16": "float16", "bf16": "bfloat16", "qi8": "int8"}


def _torch():
    import torch
    return torch


class _TorchAllocator:
    """Device memory for the library from the PyTorch caching allocator."""

    def __init__(self):
        self.live = {}
        self.alloc_cb = _sn.ALLOC_FN(self._alloc)
        self.free_cb = _sn.FREE_FN(self._free)

    def _alloc(self, nbytes, ctx):
        try:
            torch = _torch()
            t = torch.empty(int(nbytes), dtype=torch.uint8, device="cuda")
            p = t.data_ptr()
            self.live[p] = t
            return p
        except Exception:
            return None

    def _free(self, ptr, ctx):
        self.live.pop(ptr, None)


def storage_shape(shape_nchw, layout):
    n, c, h, w = shape_nchw
    return (n, c, h, w) if layout == "nchw" else (n, h, w, c)


def _stream_ptr(stream):
    torch = _torch()
    if stream is None:
        stream = torch.cuda.current_stream()
    return C.c_void_p(stream.cuda_stream)


class Graph:
    """A net (section III-B) with its routine candidates, cost table and path."""

    def __init__(self, in_shape, in_schema, out_schema, schemas, torch_alloc=True):
        self.in_shape = tuple(int(v) for v in in_shape)
        self.in_schema = tuple(in_schema)
        self.out_schema = tuple(out_schema)
        self.schemas = [tuple(s) for s in schemas]
        self._alloc = _TorchAllocator() if torch_alloc else None
        arr = (_sn.sn_schema * len(self.schemas))(*[_sn.schema(s) for s in self.schemas])
        shp = (C.c_int64 * 4)(*self.in_shape)
        h = C.c_void_p()
        a = self._alloc.alloc_cb if self._alloc else _sn.ALLOC_FN()
        f = self._alloc.free_cb if self._alloc else _sn.FREE_FN()
        check(lib().sn_graph_create(shp, _sn.schema(self.in_schema), _sn.schema(self.out_schema), arr,
                                    len(self.schemas), a, f, None, C.byref(h)))
        self.h = h
        self._last_shape = self.in_shape
        self.n_user = 0

    def __del__(self):
        h = getattr(self, "h", None)
        if h is not None and h.value:
            lib().sn_graph_destroy(h)
            self.h = None

    # ------------------------------------------------------------- building
    def add_input(self, shape):
        """Another net input (before any layer); returns its id (-2, -3, ...)."""
        shp = (C.c_int64 * 4)(*[int(v) for v in shape])
        i = C.c_int32(0)
        check(lib().sn_add_input(self.h, shp, C.byref(i)))
        return i.value

    def set_outputs(self, ids):
        """The net outputs, in order (default: the last layer added)."""
        arr = (C.c_int32 * len(ids))(*[int(v) for v in ids])
        check(lib().sn_set_outputs(self.h, arr, len(ids)))

    def io_counts(self):
        a, b = C.c_int32(0), C.c_int32(0)
        check(lib().sn_get_io(self.h, C.byref(a), C.byref(b)))
        return a.value, b.value

    def add_layer(self, type_, params=None, inputs=(-1,), weight=None, bias=None) -> int:
        ins = (C.c_int32 * len(inputs))(*inputs)
        p = None
        if type_ in (_sn.SN_L_CONV2, _sn.SN_L_DWCONV2):
            p = _sn.sn_conv_params(params["c_in"], params["c_out"], params["kh"], params["kw"],
                                   params["sh"], params["sw"], params["ph"], params["pw"],
                                   params.get("dh", 1), params.get("dw", 1), params.get("groups", 1),
                                   _sn.SN_ACT[params.get("act", "none")])
        elif type_ == _sn.SN_L_MAXPOOL:
            p = _sn.sn_pool_params(params["kh"], params["kw"], params["sh"], params["sw"], params["ph"],
                                   params["pw"])
        elif type_ in (_sn.SN_L_ADD, _sn.SN_L_MUL):
            p = _sn.sn_add_params(_sn.SN_ACT[(params or {}).get("act", "none")])
        elif type_ == _sn.SN_L_DENSE:
            p = _sn.sn_dense_params(params["in_features"], params["out_features"],
                                    _sn.SN_ACT[params.get("act", "none")])
        w = np.ascontiguousarray(weight, dtype=np.float32) if weight is not None else None
        b = np.ascontiguousarray(bias, dtype=np.float32) if bias is not None else None
        out = C.c_int32()
        check(lib().sn_add_layer(self.h, type_, C.byref(p) if p is not None else None, ins, len(inputs),
                                 w.ctypes.data if w is not None else None,
                                 b.ctypes.data if b is not None else None, C.byref(out)))
        self.n_user += 1
        return out.value

    def fuse_residual(self):
        """sn_fuse_residual: the library's residual-add fusion pass.  Returns
        (new_id, n_fused): new_id[old] = each added layer's new id (-1 for a
        conv2 folded into its add)."""
        m = self.n_user
        ids = (C.c_int32 * max(m, 1))()
        nf = C.c_int32()
        check(lib().sn_fuse_residual(self.h, ids, m, C.byref(nf)))
        new_id = [int(ids[i]) for i in range(m)]
        self.n_user = sum(1 for v in new_id if v >= 0)
        return new_id, nf.value

    # ------------------------------------------------------------ cost table
    def cost_table(self):
        t = _sn.sn_cost_table()
        check(lib().sn_get_cost_table(self.h, C.byref(t)))
        cands = (_sn.sn_candidate * t.n_candidates)()
        edges = np.zeros(2 * t.n_edges, np.int32)
        adapt = np.zeros(t.n_edges * t.n_schemas * t.n_schemas, np.int64)
        t.candidates = cands
        t.edges = edges.ctypes.data_as(C.POINTER(C.c_int32))
        t.adapt_cost = adapt.ctypes.data_as(C.POINTER(C.c_int64))
        check(lib().sn_get_cost_table(self.h, C.byref(t)))
        arr = np.array([(c.routine, c.variant, c.schema, c.layer, c.cost_ns, c.out_schema) for c in cands],
                       dtype=np.int64).reshape(-1, 6)
        return {"n_layers": t.n_layers, "n_schemas": t.n_schemas,
                "routine": arr[:, 0].astype(np.int32), "variant": arr[:, 1].astype(np.int32),
                "schema": arr[:, 2].astype(np.int32), "layer": arr[:, 3].astype(np.int32),
                "cost": arr[:, 4].copy(), "out_schema": arr[:, 5].astype(np.int32), "edges": edges.reshape(-1, 2),
                "adapt": adapt.reshape(t.n_edges, t.n_schemas, t.n_schemas)}

    def set_cost_table(self, table):
        n = len(table["cost"])
        cands = (_sn.sn_candidate * n)(*[
            _sn.sn_candidate(int(table["routine"][i]), int(table["variant"][i]), int(table["schema"][i]),
                             int(table["layer"][i]), int(table["cost"][i]),
                             int(table["out_schema"][i] if "out_schema" in table else table["schema"][i]))
            for i in range(n)])
        adapt = np.ascontiguousarray(table["adapt"], dtype=np.int64).ravel()
        t = _sn.sn_cost_table(table["n_layers"], table["n_schemas"], len(table["edges"]), n, cands, None,
                              adapt.ctypes.data_as(C.POINTER(C.c_int64)))
        check(lib().sn_set_cost_table(self.h, C.byref(t)))

    def schema_universe(self):
        n = C.c_int32()
        check(lib().sn_get_schema(self.h, 0, None, C.byref(n)))
        out = []
        for i in range(n.value):
            s = _sn.sn_schema()
            check(lib().sn_get_schema(self.h, i, C.byref(s), None))
            dt = {v: k for k, v in _sn.DTYPES.items()}[s.dtype]
            ly = {v: k for k, v in _sn.LAYOUTS.items()}[s.layout]
            out.append((dt, ly))
        return out

    def candidate_desc(self, cand):
        """Descriptor string of candidate `cand`: routine, schema, parameter values."""
        d = lib().sn_candidate_desc(self.h, int(cand))
        if d is None:
            raise _sn.SnError(_sn.SN_EINVAL, f"no candidate {cand}")
        return d.decode()

    # -------------------------------------------------------- tune and select
    def profile(self, warmup=3, iters=20, topk=2, passes=5, stream=None):
        o = _sn.sn_profile_opts(warmup, iters, topk, passes)
        check(lib().sn_profile(self.h, C.byref(o), _stream_ptr(stream)))

    def select_path(self, method=_sn.SN_SELECT_DPRS):
        t = self.cost_table()
        n = t["n_layers"]
        sch = np.zeros(n, np.int32)
        cand = np.zeros(n, np.int32)
        p = _sn.sn_path(0, n, sch.ctypes.data_as(C.POINTER(C.c_int32)), cand.ctypes.data_as(C.POINTER(C.c_int32)))
        check(lib().sn_select_path(self.h, method, C.byref(p)))
        return int(p.total_ns), sch, cand

    def set_path(self, candidates):
        c = np.ascontiguousarray(candidates, dtype=np.int32)
        check(lib().sn_set_path(self.h, c.ctypes.data_as(C.POINTER(C.c_int32)), len(c)))

    def set_option(self, opt, value):
        check(lib().sn_set_option(self.h, opt, int(value)))

    def layer_shape(self, i):
        s = (C.c_int64 * 4)()
        check(lib().sn_layer_shape(self.h, i, s))
        return tuple(s)

    def plan_stats(self, stream=None):
        """(plan operations, CUDA kernels) that one run launches."""
        ops, kern = C.c_int32(), C.c_int32()
        check(lib().sn_plan_stats(self.h, C.byref(ops), C.byref(kern), _stream_ptr(stream)))
        return ops.value, kern.value


    def plan_memory(self, stream=None):
        """(arena bytes, bytes the same activations take unshared) of the plan."""
        a, b = C.c_int64(), C.c_int64()
        check(lib().sn_plan_memory(self.h, C.byref(a), C.byref(b), _stream_ptr(stream)))
        return a.value, b.value

    def save_plan(self, path):
        check(lib().sn_save_plan(self.h, str(path).encode()))

    def load_plan(self, path):
        check(lib().sn_load_plan(self.h, str(path).encode()))

    # ------------------------------------------------------ qint8 scales
    def set_qscale(self, layer_id, scale):
        """Scale of a blob kept in qi8: layer_id from add_layer, -1 = net input."""
        check(lib().sn_set_qscale(self.h, int(layer_id), float(scale)))

    def get_qscale(self, layer_id):
        v = C.c_float(0.0)
        check(lib().sn_get_qscale(self.h, int(layer_id), C.byref(v)))
        return v.value

    def calibrate(self, x, stream=None):
        """Set every blob's qi8 scale from one float-path run on x (max |x| / 127)."""
        check(lib().sn_calibrate(self.h, C.c_void_p(x.data_ptr()), _stream_ptr(stream)))

    # --------------------------------------------------------------- running
    def output_shape(self):
        t = self.cost_table()
        return self.layer_shape(t["n_layers"] - 1)

    def new_output(self):
        torch = _torch()
        shp = storage_shape(self.output_shape(), self.out_schema[1])
        return torch.empty(shp, dtype=getattr(torch, TORCH_DTYPES[self.out_schema[0]]), device="cuda")

    def run(self, x, out=None, stream=None):
        if out is None:
            out = self.new_output()
        check(lib().sn_run(self.h, C.c_void_p(x.data_ptr()), C.c_void_p(out.data_ptr()), _stream_ptr(stream)))
        return out

    def run_host(self, x_host, out_host, stream=None):
        """sn_run_host: x_host / out_host are host tensors (pinned for asynchronous
        copies) of the input and output; the copies run inside the library, on the
        stream; synchronise the stream before reading out_host."""
        check(lib().sn_run_host(self.h, C.c_void_p(x_host.data_ptr()), C.c_void_p(out_host.data_ptr()),
                                _stream_ptr(stream)))
        return out_host

    def output_shapes(self):
        """Logical shapes of the net outputs (in order)."""
        t = self.cost_table()
        n = t["n_layers"]
        srcs = [int(t["edges"][e][0]) for e in range(len(t["edges"])) if int(t["edges"][e][1]) == n - 1]
        return [self.layer_shape(j) for j in srcs]

    def run_multi(self, xs, outs=None, stream=None):
        """Run a net with several inputs / outputs; returns the output tensors."""
        torch = _torch()
        if outs is None:
            outs = [torch.empty(storage_shape(sh, self.out_schema[1]),
                                dtype=getattr(torch, TORCH_DTYPES[self.out_schema[0]]), device="cuda")
                    for sh in self.output_shapes()]
        ins = (C.c_void_p * len(xs))(*[x.data_ptr() for x in xs])
        os_ = (C.c_void_p * len(outs))(*[o.data_ptr() for o in outs])
        check(lib().sn_run_multi(self.h, ins, len(xs), os_, len(outs), _stream_ptr(stream)))
        return outs

    def run_timed(self, x, out=None, stream=None):
        if out is None:
            out = self.new_output()
        t = self.cost_table()
        lm = np.zeros(t["n_layers"], np.float32)
        em = np.zeros(max(1, len(t["edges"])), np.float32)
        check(lib().sn_run_timed(self.h, C.c_void_p(x.data_ptr()), C.c_void_p(out.data_ptr()),
                                 _stream_ptr(stream), lm.ctypes.data_as(C.POINTER(C.c_float)),
                                 em.ctypes.data_as(C.POINTER(C.c_float))))
        return out, lm, em


def convert(x, from_schema, to_schema, shape_nchw, out=None, stream=None):
    """The adapt routine on its own: cast and/or permute a blob (bit-exact)."""
    torch = _torch()
    if out is None:
        out = torch.empty(storage_shape(shape_nchw, to_schema[1]),
                          dtype=getattr(torch, TORCH_DTYPES[to_schema[0]]), device="cuda")
    shp = (C.c_int64 * 4)(*shape_nchw)
    check(lib().sn_convert(C.c_void_p(x.data_ptr()), _sn.schema(from_schema), C.c_void_p(out.data_ptr()),
                           _sn.schema(to_schema), shp, _stream_ptr(stream)))
    return out


def convert_q(x, from_schema, to_schema, shape_nchw, qscale, out=None, stream=None):
    """The adapt routine with a qi8 side: quantise, dequantise or permute codes."""
    torch = _torch()
    if out is None:
        out = torch.empty(storage_shape(shape_nchw, to_schema[1]),
                          dtype=getattr(torch, TORCH_DTYPES[to_schema[0]]), device="cuda")
    shp = (C.c_int64 * 4)(*shape_nchw)
    check(lib().sn_convert_q(C.c_void_p(x.data_ptr()), _sn.schema(from_schema), C.c_void_p(out.data_ptr()),
                             _sn.schema(to_schema), shp, C.c_float(qscale), _stream_ptr(stream)))
    return out
