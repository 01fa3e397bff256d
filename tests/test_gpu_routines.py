"""Per-routine parity on the GPU through the C ABI: every routine of every
layer type, in every schema it serves, against the oracle on the same stored
inputs.  Adapt conversions are checked bit for bit."""
import zlib

import numpy as np
import pytest

import oracle
import synth
from oracle.net import run_layer, run_net
from paper_2110_06037_gb300 import build_graph, convert

from gpu_helpers import TOL, find_candidate, from_device, maxrel, raw_bits, stored_values, to_device

pytestmark = pytest.mark.gpu

DTS = ("f32", "f16", "bf16")
LAYS = ("nchw", "nhwc")
SCHEMAS = [(d, l) for d in DTS for l in LAYS]


def run_one(layer, x, schema, routine, variant):
    """Build a one-layer net in `schema`, force (routine, variant), run, return fp64 NCHW."""
    import torch
    spec = dict(layer)
    spec["inputs"] = [-1] * (2 if layer["type"] == "add" else 1)
    g = build_graph([spec], x.shape, schema, schema, [schema])
    t = g.cost_table()
    c = find_candidate(t, 1, routine, variant, 0)
    if c is None:
        return None
    cands = [int(np.flatnonzero(t["layer"] == 0)[0]), c, int(np.flatnonzero(t["layer"] == 2)[0])]
    g.set_path(cands)
    xd = to_device(x, schema)
    y = g.run(xd)
    torch.cuda.synchronize()
    return from_device(y, schema)


def ref_one(layer, x, dt):
    xs = stored_values(x, dt)
    ins = [xs, xs] if layer["type"] == "add" else [xs]
    return run_layer(layer, ins, dt)


CONV_CASES = [
    # N, C, H, W, K, k, s, p, d, groups
    (1, 3, 32, 32, 16, 3, 1, 1, 1, 1),
    (1, 16, 32, 32, 32, 3, 2, 1, 1, 1),
    (2, 24, 9, 11, 40, 3, 1, 1, 1, 1),     # ragged tiles
    (1, 64, 14, 14, 64, 1, 1, 0, 1, 1),
    (2, 32, 7, 7, 48, 1, 2, 0, 1, 1),
    (1, 8, 10, 10, 8, 3, 1, 1, 1, 2),      # groups
    (1, 3, 23, 23, 16, 7, 2, 3, 1, 1),     # stem-like 7x7 s2
    (1, 8, 12, 12, 8, 3, 1, 2, 2, 1),      # dilation
    (1, 130, 5, 5, 66, 3, 1, 1, 1, 1),     # channels past a tile edge
    (1, 16, 1, 1, 8, 3, 1, 1, 1, 1),       # 1x1 image, 3x3 kernel (padding only)
    (2, 3, 30, 30, 64, 7, 2, 3, 1, 1),     # the ResNet stem's shape class (space-to-depth routine)
    (1, 4, 17, 19, 24, 3, 2, 1, 1, 1),     # space-to-depth: 4 channels, odd extents
    (1, 2, 16, 16, 8, 5, 2, 2, 1, 1),      # space-to-depth: 5x5 kernel
]
ROUTINES = ([("conv2/direct", 0), ("conv2/igemm_simt", 0), ("conv2/igemm_simt", 1), ("conv2/wino_f2x2_3x3", 0),
             ("conv2/wino_f4x4_3x3", 0), ("conv2/wino_f6x6_3x3", 0)]
            + [("conv2/igemm_tc", v) for v in range(6)] + [("conv2/im2col_tc", v) for v in range(3)]
            + [("conv2/s2d_tc", v) for v in range(4)])


@pytest.mark.parametrize("case", CONV_CASES)
@pytest.mark.parametrize("schema", SCHEMAS)
def test_conv_routines(case, schema):
    N, C, H, W, K, k, s, p, d, g = case
    rng = np.random.default_rng(zlib.crc32(repr((case, schema)).encode()))
    x = rng.standard_normal((N, C, H, W)).astype(np.float32)
    layer = synth.conv(C, K, k, s, p, act="relu", groups=g, d=d)
    layer["weight"] = (rng.standard_normal((K, C // g, k, k)) * np.sqrt(2.0 / (C // g * k * k))).astype(np.float32)
    layer["bias"] = (rng.standard_normal(K) * 0.1).astype(np.float32)
    ref = ref_one(layer, x, schema[0])
    ran = 0
    for rname, v in ROUTINES:
        got = run_one(layer, x, schema, rname, v)
        if got is None:
            continue
        ran += 1
        err = maxrel(got, ref)
        assert err <= TOL[schema[0]], (rname, v, err)
    assert ran >= 1


DW_CASES = [(1, 32, 16, 16, 1), (2, 24, 9, 9, 2), (1, 144, 28, 28, 1), (1, 40, 7, 7, 2), (1, 8, 1, 1, 1),
            (2, 576, 14, 14, 1),    # channel slices of 192 (TMA box limit 256)
            (4, 320, 9, 9, 1),      # two slices of 160, ragged column blocks
            (3, 96, 30, 30, 2),
            (16, 64, 57, 57, 2),    # odd extent, stride 2, ranges spanning images
            (48, 128, 48, 48, 1)]   # ranges longer than the row ring (slots reused)


@pytest.mark.parametrize("case", DW_CASES)
@pytest.mark.parametrize("schema", SCHEMAS)
def test_depthwise(case, schema):
    N, C, H, W, s = case
    rng = np.random.default_rng(zlib.crc32(repr((case, schema)).encode()))
    x = rng.standard_normal((N, C, H, W)).astype(np.float32)
    layer = synth.dwconv(C, 3, s, act="relu6")
    layer["weight"] = (rng.standard_normal((C, 1, 3, 3)) * np.sqrt(2 / 9)).astype(np.float32)
    layer["bias"] = (rng.standard_normal(C) * 0.1).astype(np.float32)
    ref = ref_one(layer, x, schema[0])
    outs = {}
    # routine parameters: register window / rows in shared memory / (small maps)
    # band tiles in shared memory (NHWC); row / plane tile (NCHW)
    variants = (0, 1, 2) if schema[1] == "nhwc" else (0, 1)
    for v in variants:
        got = run_one(layer, x, schema, "dwconv2/direct", v)
        if got is None:  # the band kernel does not apply to this map (a 3-row band would not fit)
            assert v == 2 and W > 110
            continue
        assert maxrel(got, ref) <= TOL[schema[0]], v
        outs[v] = got
    if schema[1] == "nhwc":
        # the NHWC kernels accumulate the nine taps in the same order (bias,
        # then rows, then columns): in f32 with exact products for bf16, in
        # packed half2 for f16: equal results (the f32 ring fallback differs)
        if schema[0] != "f32":
            assert np.array_equal(outs[0], outs[1])
        if 2 in outs:
            assert np.array_equal(outs[0], outs[2])


@pytest.mark.parametrize("schema", SCHEMAS)
def test_pool_gap_add_dense(schema):
    rng = np.random.default_rng(3)
    x = rng.standard_normal((2, 16, 13, 11)).astype(np.float32)
    mp = synth.maxpool(3, 2, 1)
    got = run_one(mp, x, schema, "maxpool/direct", 0)
    # max pooling selects a stored value: exact
    assert np.array_equal(got, ref_one(mp, x, schema[0]))
    gp = synth.gap()
    assert maxrel(run_one(gp, x, schema, "gap/reduce", 0), ref_one(gp, x, schema[0])) <= TOL[schema[0]]
    ad = synth.add(act="relu")
    assert maxrel(run_one(ad, x, schema, "add/eltwise", 0), ref_one(ad, x, schema[0])) <= TOL[schema[0]]
    xd = rng.standard_normal((3, 70, 1, 1)).astype(np.float32)
    de = synth.dense(70, 33)
    de["weight"] = (rng.standard_normal((33, 70)) * 0.2).astype(np.float32)
    de["bias"] = (rng.standard_normal(33) * 0.1).astype(np.float32)
    assert maxrel(run_one(de, xd, schema, "dense/simt", 0), ref_one(de, xd, schema[0])) <= TOL[schema[0]]
    # dense childnet on the tensor-core GEMM (fp16/bf16 only)
    xd = rng.standard_normal((5, 64, 1, 1)).astype(np.float32)
    de = synth.dense(64, 40)
    de["weight"] = (rng.standard_normal((40, 64)) * 0.2).astype(np.float32)
    de["bias"] = (rng.standard_normal(40) * 0.1).astype(np.float32)
    ref = ref_one(de, xd, schema[0])
    for v in range(3):
        got = run_one(de, xd, schema, "dense/gemm_tc", v)
        if got is not None:
            assert schema[0] != "f32"
            assert maxrel(got, ref) <= TOL[schema[0]], v


@pytest.mark.parametrize("shape", [(2, 16, 13, 11), (1, 40, 7, 7), (3, 12, 5, 5)])
@pytest.mark.parametrize("schema", SCHEMAS)
def test_mul_squeeze_excite_scale(shape, schema):
    """gap -> per-channel scale of the same blob (+ hard swish): the vector NHWC
    kernel (C * elem a multiple of 16 bytes), the element kernel otherwise."""
    import torch
    rng = np.random.default_rng(zlib.crc32(repr((shape, schema, "mul")).encode()))
    x = (rng.standard_normal(shape) * 2).astype(np.float32)
    net = [dict(synth.gap(), inputs=[-1]), dict(synth.mul(act="hswish"), inputs=[-1, 0])]
    ref = run_net(net, x, schema[0])
    g = build_graph(net, x.shape, schema, schema, [schema])
    t = g.cost_table()
    pc = [int(np.flatnonzero(t["layer"] == 0)[0]), find_candidate(t, 1, "gap/reduce", 0, 0),
          find_candidate(t, 2, "mul/eltwise", 0, 0), int(np.flatnonzero(t["layer"] == 3)[0])]
    g.set_path(pc)
    y = g.run(to_device(x, schema))
    torch.cuda.synchronize()
    assert maxrel(from_device(y, schema), ref) <= TOL[schema[0]]


@pytest.mark.parametrize("act", ["hswish", "hsigmoid"])
@pytest.mark.parametrize("schema", [("f32", "nchw"), ("f16", "nhwc"), ("bf16", "nhwc")])
def test_conv_hard_activations(act, schema):
    """MobileNetV3's activations in the epilogues of every conv routine the
    layer offers (direct, SIMT GEMM, Winograd, tensor cores)."""
    import torch
    rng = np.random.default_rng(zlib.crc32(repr((act, schema)).encode()))
    x = (rng.standard_normal((2, 32, 9, 9)) * 2).astype(np.float32)
    layer = synth.conv(32, 64, 3, 1, 1, act=act)
    layer["weight"] = (rng.standard_normal((64, 32, 3, 3)) * np.sqrt(2 / 288)).astype(np.float32)
    layer["bias"] = (rng.standard_normal(64) * 0.5).astype(np.float32)
    ref = ref_one(layer, x, schema[0])
    g = build_graph([dict(layer, inputs=[-1])], x.shape, schema, schema, [schema])
    t = g.cost_table()
    io = [int(np.flatnonzero(t["layer"] == 0)[0]), int(np.flatnonzero(t["layer"] == 2)[0])]
    ran = 0
    for c in np.flatnonzero(t["layer"] == 1):
        g.set_path([io[0], int(c), io[1]])
        y = g.run(to_device(x, schema))
        torch.cuda.synchronize()
        assert maxrel(from_device(y, schema), ref) <= TOL[schema[0]], int(t["routine"][c])
        ran += 1
    assert ran >= 2


# planes of 196 (8-byte bf16 rows, 16-byte f32 rows), 49 (element-wide rows),
# 81 and 60 (ragged tiles per image) and 130 channels (ragged tiles on both
# axes, element-wide channel rows)
CONVERT_SHAPES = [(2, 5, 7, 9), (1, 64, 56, 56), (3, 130, 1, 1), (1, 3, 65, 67), (2, 24, 14, 14),
                  (2, 40, 7, 7), (2, 130, 14, 14), (1, 1024, 14, 14), (5, 64, 9, 9), (4, 256, 14, 14),
                  (3, 72, 10, 6)]


@pytest.mark.parametrize("shape", CONVERT_SHAPES)
def test_convert_bit_exact(shape):
    import torch
    rng = np.random.default_rng(11)
    x = (rng.standard_normal(shape) * 3).astype(np.float32)
    flat = x.reshape(-1)
    flat[: min(6, flat.size)] = np.array([7e4, -1e5, 3e-8, -6e-6, 65520.0, 0.0], np.float32)[: min(6, flat.size)]
    for d_in in DTS:
        for l_in in LAYS:
            xd = to_device(x, (d_in, l_in))
            vin = stored_values(x, d_in).astype(np.float32)
            for d_out in DTS:
                for l_out in LAYS:
                    y = convert(xd, (d_in, l_in), (d_out, l_out), shape)
                    torch.cuda.synchronize()
                    ref = oracle.to_bits(vin, d_out)
                    if l_out == "nhwc":
                        ref = oracle.nchw_to_nhwc(ref)
                    got = raw_bits(y).reshape(ref.shape)
                    assert np.array_equal(got, ref.view(got.dtype)), (d_in, l_in, d_out, l_out)


def test_convert_empty_is_noop():
    import torch
    x = torch.zeros(4, device="cuda")
    convert(x, ("f32", "nchw"), ("f16", "nhwc"), (0, 3, 4, 4), out=torch.zeros(1, device="cuda", dtype=torch.float16))


RES_CASES = [
    # N, C, H, W, k, p  (C -> C channels, stride 1, "same" padding: the output has the input's shape)
    (2, 24, 9, 11, 3, 1),     # C not a multiple of 64
    (1, 64, 14, 14, 1, 0),    # plain GEMM tile
    (2, 128, 8, 8, 3, 1),     # CTA pairs, two channel blocks per stage
    (2, 256, 7, 7, 3, 1),     # K-split variants: the residual is added by the reduction
    (4, 512, 7, 7, 1, 0),     # plain GEMM K split
]


@pytest.mark.parametrize("case", RES_CASES)
@pytest.mark.parametrize("schema", SCHEMAS)
def test_conv_residual(case, schema):
    """conv2 with a residual input (a fused add): y = relu(conv(x) + b + r),
    r = the 3x3 stride-1 max pool of x (a blob distinct from the conv input),
    for every direct and tensor-core routine parameter the layer offers."""
    import torch
    N, C, H, W, k, p = case
    rng = np.random.default_rng(zlib.crc32(repr((case, schema, "res")).encode()))
    x = rng.standard_normal((N, C, H, W)).astype(np.float32)
    pool = {"type": "maxpool", "name": "pool", "inputs": [-1],
            "params": dict(kh=3, kw=3, sh=1, sw=1, ph=1, pw=1)}
    conv = synth.conv(C, C, k, 1, p, act="relu")
    conv["weight"] = (rng.standard_normal((C, C, k, k)) * np.sqrt(2.0 / (C * k * k))).astype(np.float32)
    conv["bias"] = (rng.standard_normal(C) * 0.1).astype(np.float32)
    conv["inputs"] = [-1, 0]
    net = [pool, conv]
    dt = schema[0]
    xs = stored_values(x, dt)
    r = run_layer(pool, [xs], dt)
    ref = run_layer(conv, [xs, r], dt)
    g = build_graph(net, x.shape, schema, schema, [schema])
    t = g.cost_table()
    io_in = int(np.flatnonzero(t["layer"] == 0)[0])
    io_out = int(np.flatnonzero(t["layer"] == 3)[0])
    pc = find_candidate(t, 1, "maxpool/direct", 0, 0)
    ran = 0
    for c in range(len(t["cost"])):
        if t["layer"][c] != 2:
            continue
        g.set_path([io_in, pc, c, io_out])
        y = g.run(to_device(x, schema))
        torch.cuda.synchronize()
        err = maxrel(from_device(y, schema), ref)
        assert err <= TOL[dt], (int(t["routine"][c]), int(t["variant"][c]), err)
        ran += 1
    assert ran >= 1
