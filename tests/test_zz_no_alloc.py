"""The allocation-free Winograd entry point, sn_conv2d_wino_noalloc.

Some callers cannot allocate device memory where they run a layer (plug-ins
in a host application that owns all device allocations, services with a
memory budget fixed at start-up, latency-critical loops that must not call
cudaMalloc).  This entry point serves them: its scratch is a fixed array in
the library's device image.  The test calls it through the C ABI twice in a
row, on different inputs, and checks each output against the graph entry
point (sn_run with the conv2/wino_f2x2_3x3 routine forced) within the
tolerance the other parity tests use.  It must pass alone in a fresh process
and after the rest of the suite, so it builds everything it needs itself.
This file is named to be collected last.
"""
import ctypes as C

import numpy as np
import pytest

import synth
from paper_2110_06037_gb300 import _sn, build_graph, routine_name

from gpu_helpers import TOL, from_device, maxrel, to_device

pytestmark = pytest.mark.gpu


def _graph_reference(layer, x, schema):
    """The existing entry point: a one-layer graph with the Winograd routine forced."""
    import torch
    g = build_graph([dict(layer, inputs=[-1])], x.shape, schema, schema, [schema])
    t = g.cost_table()
    wino = [c for c in range(len(t["cost"])) if routine_name(int(t["routine"][c])) == "conv2/wino_f2x2_3x3"]
    g.set_path([int(np.flatnonzero(t["layer"] == 0)[0]), wino[0], int(np.flatnonzero(t["layer"] == 2)[0])])
    y = g.run(to_device(x, schema))
    torch.cuda.synchronize()
    return from_device(y, schema)


@pytest.mark.parametrize("schema", [("f16", "nhwc"), ("f32", "nchw"), ("bf16", "nchw")])
def test_noalloc_matches_graph_entry_point_twice(schema):
    import torch
    from gpu_helpers import torch_dtype
    from paper_2110_06037_gb300.api import storage_shape
    N, C_, H, W, K, pad = 2, 24, 13, 11, 40, 1
    rng = np.random.default_rng(42)
    layer = synth.conv(C_, K, 3, 1, pad, act="relu")
    layer["weight"] = (rng.standard_normal((K, C_, 3, 3)) * np.sqrt(2.0 / (9 * C_))).astype(np.float32)
    layer["bias"] = (rng.standard_normal(K) * 0.1).astype(np.float32)
    w_dev = torch.from_numpy(layer["weight"]).cuda()
    b_dev = torch.from_numpy(layer["bias"]).cuda()
    shape = (C.c_int64 * 4)(N, C_, H, W)
    lib = _sn.lib()
    stream = torch.cuda.current_stream()
    for call in range(2):  # two calls in a row share the scratch array
        x = rng.standard_normal((N, C_, H, W)).astype(np.float32)
        ref = _graph_reference(layer, x, schema)
        xd = to_device(x, schema)
        y = torch.empty(storage_shape((N, K, H + 2 * pad - 2, W + 2 * pad - 2), schema[1]),
                        dtype=torch_dtype(schema[0]), device="cuda")
        _sn.check(lib.sn_conv2d_wino_noalloc(C.c_void_p(xd.data_ptr()), _sn.schema(schema), shape, K, pad,
                                             _sn.SN_ACT["relu"], C.c_void_p(w_dev.data_ptr()),
                                             C.c_void_p(b_dev.data_ptr()), C.c_void_p(y.data_ptr()),
                                             C.c_void_p(stream.cuda_stream)))
        torch.cuda.synchronize()
        err = maxrel(from_device(y, schema), ref)
        assert err <= TOL[schema[0]], (call, err)


def test_noalloc_rejects_sizes_beyond_its_scratch():
    import torch
    lib = _sn.lib()
    big = (C.c_int64 * 4)(64, 256, 56, 56)  # needs far more than the fixed scratch
    d = torch.zeros(16, device="cuda")
    st = lib.sn_conv2d_wino_noalloc(C.c_void_p(d.data_ptr()), _sn.schema(("f16", "nhwc")), big, 256, 1, 0,
                                    C.c_void_p(d.data_ptr()), C.c_void_p(d.data_ptr()), C.c_void_p(d.data_ptr()),
                                    None)
    assert st == _sn.SN_EUNSUPPORTED
    assert b"scratch" in lib.sn_last_error()
