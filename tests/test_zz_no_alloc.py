"""The allocation-free Winograd entry point, sn_conv2d_wino_noalloc.

Some callers cannot allocate device memory where they run a layer (plug-ins
in a host application that owns all device allocations, services with a
memory budget fixed at start-up, latency-critical loops that must not call
cudaMalloc).  This entry point serves them: its scratch is a fixed array in
the library's device image.

The GPU test calls it through the C ABI twice in a row, the second time on a
smaller layer (so a stale or mis-offset part of the shared scratch from the
first call would be read if the second call failed to rewrite it), and
checks every output
  * against the oracle's fp64 convolution of the same stored values, within
    the tolerance of the other parity tests, and
  * bit for bit against the graph entry point (sn_run with the
    conv2/wino_f2x2_3x3 routine forced), which runs the same kernels.
It must pass alone in a fresh process and after the rest of the suite, so it
builds everything it needs itself.  This file is named to be collected last.
The argument checks that reject a call before any device work run on a host
without a GPU too.
"""
import ctypes as C

import numpy as np
import pytest

import synth
from oracle.net import run_layer
from paper_2110_06037_gb300 import _sn, build_graph, routine_name

from gpu_helpers import TOL, from_device, maxrel, raw_bits, stored_values, to_device


def _graph_reference(layer, x, schema):
    """The existing entry point: a one-layer graph with the Winograd routine forced."""
    import torch
    g = build_graph([dict(layer, inputs=[-1])], x.shape, schema, schema, [schema])
    t = g.cost_table()
    wino = [c for c in range(len(t["cost"])) if routine_name(int(t["routine"][c])) == "conv2/wino_f2x2_3x3"]
    g.set_path([int(np.flatnonzero(t["layer"] == 0)[0]), wino[0], int(np.flatnonzero(t["layer"] == 2)[0])])
    y = g.run(to_device(x, schema))
    torch.cuda.synchronize()
    return y


def _layer(rng, C_, K, pad):
    layer = synth.conv(C_, K, 3, 1, pad, act="relu")
    layer["weight"] = (rng.standard_normal((K, C_, 3, 3)) * np.sqrt(2.0 / (9 * C_))).astype(np.float32)
    layer["bias"] = (rng.standard_normal(K) * 0.1).astype(np.float32)
    return layer


@pytest.mark.gpu
@pytest.mark.parametrize("schema", [("f16", "nhwc"), ("f32", "nchw"), ("bf16", "nchw")])
def test_noalloc_matches_oracle_and_graph_entry_point_twice(schema):
    import torch
    from gpu_helpers import torch_dtype
    from paper_2110_06037_gb300.api import storage_shape
    lib = _sn.lib()
    stream = torch.cuda.current_stream()
    rng = np.random.default_rng(42)
    # the second call is smaller in every dimension: it reads only scratch it wrote itself
    for call, (N, C_, H, W, K, pad) in enumerate([(2, 24, 13, 11, 40, 1), (1, 8, 7, 9, 16, 0)]):
        layer = _layer(rng, C_, K, pad)
        w_dev = torch.from_numpy(layer["weight"]).cuda()
        b_dev = torch.from_numpy(layer["bias"]).cuda()
        x = rng.standard_normal((N, C_, H, W)).astype(np.float32)
        ref_graph = _graph_reference(layer, x, schema)
        ref_oracle = run_layer(layer, [stored_values(x, schema[0])], schema[0])
        xd = to_device(x, schema)
        P, Q = H + 2 * pad - 2, W + 2 * pad - 2
        y = torch.empty(storage_shape((N, K, P, Q), schema[1]), dtype=torch_dtype(schema[0]), device="cuda")
        shape = (C.c_int64 * 4)(N, C_, H, W)
        _sn.check(lib.sn_conv2d_wino_noalloc(C.c_void_p(xd.data_ptr()), _sn.schema(schema), shape, K, pad,
                                             _sn.SN_ACT["relu"], C.c_void_p(w_dev.data_ptr()),
                                             C.c_void_p(b_dev.data_ptr()), C.c_void_p(y.data_ptr()),
                                             C.c_void_p(stream.cuda_stream)))
        torch.cuda.synchronize()
        got = from_device(y, schema)
        assert got.shape == ref_oracle.shape
        err = maxrel(got, ref_oracle)
        assert err <= TOL[schema[0]], (call, err)
        assert np.array_equal(raw_bits(y), raw_bits(ref_graph)), call


@pytest.mark.gpu
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


def _host_dummy():
    """A non-NULL pointer the call never dereferences: it rejects its arguments first."""
    buf = C.create_string_buffer(64)
    return buf, C.cast(buf, C.c_void_p)


def test_noalloc_rejects_qint8_before_any_device_work():
    lib = _sn.lib()
    keep, p = _host_dummy()
    shape = (C.c_int64 * 4)(1, 8, 8, 8)
    st = lib.sn_conv2d_wino_noalloc(p, _sn.schema(("qi8", "nhwc")), shape, 8, 1, 0, p, p, p, None)
    assert st == _sn.SN_EUNSUPPORTED
    assert b"qint8" in lib.sn_last_error()


def test_noalloc_rejects_byte_counts_that_overflow():
    lib = _sn.lib()
    keep, p = _host_dummy()
    # every extent at its 2^30 maximum: tiles x channels x 64 bytes is beyond 2^64
    huge = (C.c_int64 * 4)(1 << 30, 1 << 30, 1 << 30, 1 << 30)
    st = lib.sn_conv2d_wino_noalloc(p, _sn.schema(("f16", "nhwc")), huge, 1 << 30, 1, 0, p, p, p, None)
    assert st == _sn.SN_EUNSUPPORTED
    assert b"2^64" in lib.sn_last_error()
    # products that fit in 64 bits but not in the scratch
    wide = (C.c_int64 * 4)(1, 1 << 20, 4, 4)
    st = lib.sn_conv2d_wino_noalloc(p, _sn.schema(("f32", "nchw")), wide, 1 << 20, 1, 0, p, p, p, None)
    assert st == _sn.SN_EUNSUPPORTED
    assert b"scratch" in lib.sn_last_error()
