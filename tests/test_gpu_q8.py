"""qint8 schema on the GPU through the C ABI (section II-C quantisation,
hybrid tuning of section V-C): the quantise / dequantise / permute adapts,
every qint8 routine, a whole net kept in qint8, calibration, and DPRS over a
float and a qint8 schema.  Codes must equal the oracle's bit for bit."""
import zlib

import numpy as np
import pytest

import oracle
from oracle import q8
from oracle.net import run_net
from paper_2110_06037_gb300 import build_graph, convert_q, routine_name

from gpu_helpers import from_device, maxrel, raw_bits, stored_values, to_device

pytestmark = pytest.mark.gpu

F32 = np.float32


def codes_to_device(q_nchw, lay):
    import torch
    q = np.asarray(q_nchw, np.int8)
    if lay == "nhwc":
        q = oracle.nchw_to_nhwc(q)
    return torch.from_numpy(np.ascontiguousarray(q)).cuda()


def codes_from_device(t, lay):
    a = t.detach().cpu().numpy().astype(np.int8)
    return oracle.nhwc_to_nchw(a) if lay == "nhwc" else a


# ------------------------------------------------------------------ adapts
SHAPES = [(2, 5, 7, 3), (1, 64, 8, 8), (3, 1, 4, 4), (1, 3, 1, 1), (2, 33, 5, 9)]


@pytest.mark.parametrize("dt", ["f32", "f16", "bf16"])
@pytest.mark.parametrize("lay_in,lay_out", [("nchw", "nchw"), ("nhwc", "nhwc"), ("nchw", "nhwc"), ("nhwc", "nchw")])
def test_quantise_adapt(dt, lay_in, lay_out):
    rng = np.random.default_rng(zlib.crc32(f"{dt}{lay_in}{lay_out}".encode()))
    for shp in SHAPES:
        x = (3 * rng.standard_normal(shp)).astype(F32)
        s = F32(0.0371)
        want = q8.quantize(stored_values(x, dt).astype(F32), s)
        got = convert_q(to_device(x, (dt, lay_in)), (dt, lay_in), ("qi8", lay_out), shp, float(s))
        assert np.array_equal(codes_from_device(got, lay_out), want), shp


@pytest.mark.parametrize("dt", ["f32", "f16", "bf16"])
@pytest.mark.parametrize("lay_in,lay_out", [("nchw", "nchw"), ("nchw", "nhwc"), ("nhwc", "nchw")])
def test_dequantise_adapt(dt, lay_in, lay_out):
    rng = np.random.default_rng(7)
    for shp in SHAPES:
        q = rng.integers(-127, 128, shp).astype(np.int8)
        s = F32(0.173)
        want = oracle.to_bits(q8.dequantize(q, s), dt)
        if dt == "f32":
            want = want.view(np.uint32)
        got = convert_q(codes_to_device(q, lay_in), ("qi8", lay_in), (dt, lay_out), shp, float(s))
        g = raw_bits(got)
        if lay_out == "nhwc":
            g = oracle.nhwc_to_nchw(g)
        assert np.array_equal(g, want), shp


def test_code_permutation_is_exact():
    rng = np.random.default_rng(8)
    for shp in SHAPES:
        q = rng.integers(-127, 128, shp).astype(np.int8)
        got = convert_q(codes_to_device(q, "nchw"), ("qi8", "nchw"), ("qi8", "nhwc"), shp, 0.5)
        assert np.array_equal(codes_from_device(got, "nhwc"), q)


# ----------------------------------------------------------------- routines
def _force(g, t, prefer):
    """Per layer the first candidate whose routine name is in `prefer` (in
    order), else the layer's first candidate."""
    n = int(t["n_layers"])
    cands = []
    for i in range(n):
        idx = np.flatnonzero(t["layer"] == i)
        pick = int(idx[0])
        for name in prefer:
            hit = [int(c) for c in idx if routine_name(int(t["routine"][c])) == name]
            if hit:
                pick = hit[0]
                break
        cands.append(pick)
    g.set_path(cands)
    return [routine_name(int(t["routine"][c])) for c in cands]


def _ref_codes(layers, q_in, s_in, scales):
    outs = []
    for i, layer in enumerate(layers):
        ins = [q_in if j < 0 else outs[j] for j in layer["inputs"]]
        s_ins = [s_in if j < 0 else scales[j] for j in layer["inputs"]]
        outs.append(q8.run_layer(layer, ins, s_ins, scales[i]))
    return outs[-1]


def _out_scales(layers, q_in, s_in):
    """Output scales from the fp64 float net on the dequantised input."""
    _, outs = run_net(layers, q8.dequantize(q_in, s_in), keep=True)
    return [q8.absmax_scale(o.astype(F32)) for o in outs]


def run_q8(layers, q_in, s_in, scales, lay, prefer):
    import torch
    g = build_graph(layers, q_in.shape, ("qi8", lay), ("qi8", lay), [("qi8", lay)])
    g.set_qscale(-1, float(s_in))
    for i, s in enumerate(scales):
        g.set_qscale(i, float(s))
    used = _force(g, g.cost_table(), prefer)
    y = g.run(codes_to_device(q_in, lay))
    torch.cuda.synchronize()
    return codes_from_device(y, lay), used


def conv_layer(rng, c, k, ks, st, pad, dil=1, groups=1, act="relu", resid=False, dw=False):
    return {"type": "dwconv2" if dw else "conv2", "inputs": [-1, -1] if resid else [-1],
            "params": dict(c_in=c, c_out=k, kh=ks, kw=ks, sh=st, sw=st, ph=pad, pw=pad, dh=dil, dw=dil,
                           groups=c if dw else groups, act=act),
            "weight": (rng.standard_normal((k, 1 if dw else c // groups, ks, ks)) / np.sqrt(c * ks * ks / groups))
            .astype(F32),
            "bias": (0.1 * rng.standard_normal(k)).astype(F32)}


CONV_CASES = [
    # N, C, H, W, K, k, s, p, d, groups, act, residual
    (2, 8, 9, 11, 12, 3, 1, 1, 1, 1, "relu", False),
    (1, 36, 14, 14, 68, 3, 2, 1, 1, 1, "none", False),
    (2, 64, 7, 7, 64, 1, 1, 0, 1, 1, "relu", True),
    (1, 12, 12, 12, 8, 3, 1, 2, 2, 1, "relu6", False),
    (1, 3, 23, 23, 16, 7, 2, 3, 1, 1, "relu", False),   # C % 4 != 0: direct only
    (1, 8, 10, 10, 8, 3, 1, 1, 1, 2, "hswish", False),   # groups: direct only
    (3, 128, 5, 5, 132, 3, 1, 1, 1, 1, "relu", False),   # several 32-channel chunks, K past a tile
]


@pytest.mark.parametrize("case", CONV_CASES)
@pytest.mark.parametrize("routine", ["conv2/direct", "conv2/igemm_dp4a"])
@pytest.mark.parametrize("lay", ["nchw", "nhwc"])
def test_q8_conv(case, routine, lay):
    n, c, h, w, k, ks, st, pad, dil, groups, act, resid = case
    if routine == "conv2/igemm_dp4a" and (lay == "nchw" or c % 4 or k % 4 or groups != 1):
        pytest.skip("the dp4a routine serves NHWC, groups 1, C and K multiples of 4")
    rng = np.random.default_rng(zlib.crc32(repr(case).encode()))
    layer = conv_layer(rng, c, k, ks, st, pad, dil, groups, act, resid)
    q_in = rng.integers(-127, 128, (n, c, h, w)).astype(np.int8)
    s_in = F32(0.021)
    scales = _out_scales([layer], q_in, s_in)
    got, used = run_q8([layer], q_in, s_in, scales, lay, [routine])
    assert used[1] == routine
    want = _ref_codes([layer], q_in, s_in, scales)
    assert np.array_equal(got, want)
    assert np.abs(want.astype(int)).max() > 60  # the scale uses the code range


@pytest.mark.parametrize("lay", ["nchw", "nhwc"])
def test_q8_depthwise(lay):
    rng = np.random.default_rng(21)
    for (c, h, w, ks, st) in [(32, 13, 11, 3, 1), (24, 14, 14, 3, 2), (16, 9, 9, 5, 2)]:
        layer = conv_layer(rng, c, c, ks, st, ks // 2, act="relu6", dw=True)
        q_in = rng.integers(-127, 128, (2, c, h, w)).astype(np.int8)
        s_in = F32(0.05)
        scales = _out_scales([layer], q_in, s_in)
        got, used = run_q8([layer], q_in, s_in, scales, lay, ["dwconv2/direct"])
        assert used[1] == "dwconv2/direct"
        assert np.array_equal(got, _ref_codes([layer], q_in, s_in, scales))


@pytest.mark.parametrize("lay", ["nchw", "nhwc"])
def test_q8_pool_gap_add_mul(lay):
    rng = np.random.default_rng(31)
    q_in = rng.integers(-127, 128, (2, 24, 13, 15)).astype(np.int8)
    s_in = F32(0.03)
    nets = [
        [{"type": "maxpool", "inputs": [-1], "params": dict(kh=3, kw=3, sh=2, sw=2, ph=1, pw=1)}],
        [{"type": "maxpool", "inputs": [-1], "params": dict(kh=2, kw=2, sh=2, sw=2, ph=0, pw=0)}],
        [{"type": "gap", "inputs": [-1]}],
        [{"type": "add", "inputs": [-1, -1], "params": dict(act="relu")}],
        [{"type": "gap", "inputs": [-1]},
         {"type": "mul", "inputs": [-1, 0], "params": dict(act="none")}],
    ]
    for layers in nets:
        scales = _out_scales(layers, q_in, s_in)
        if layers[0]["type"] == "maxpool":
            scales = [F32(s_in * 1.5)]  # a different output scale: the maximum is requantised
        got, _ = run_q8(layers, q_in, s_in, scales, lay, [])
        want = _ref_codes(layers, q_in, s_in, scales)
        assert np.array_equal(got, want), layers[-1]["type"]


@pytest.mark.parametrize("n,i,o", [(1, 4096, 1000), (3, 2048, 40), (9, 100, 37), (32, 512, 10)])
def test_q8_dense(n, i, o):
    rng = np.random.default_rng(n * 1000 + i)
    layer = {"type": "dense", "inputs": [-1], "params": dict(in_features=i, out_features=o, act="relu"),
             "weight": (rng.standard_normal((o, i)) / np.sqrt(i)).astype(F32),
             "bias": (0.1 * rng.standard_normal(o)).astype(F32)}
    q_in = rng.integers(-127, 128, (n, i, 1, 1)).astype(np.int8)
    s_in = F32(0.01)
    scales = _out_scales([layer], q_in, s_in)
    got, used = run_q8([layer], q_in, s_in, scales, "nhwc", ["dense/simt"])
    assert used[1] == "dense/simt"
    assert np.array_equal(got, _ref_codes([layer], q_in, s_in, scales))


# ---------------------------------------------------------------- whole nets
def small_net(rng):
    """Stem (3 channels), 3x3 convs, a residual conv, max pool, depthwise,
    global pool, dense: every qint8 routine on one path."""
    return [
        conv_layer(rng, 3, 16, 3, 1, 1),                                       # 0
        dict(conv_layer(rng, 16, 16, 3, 1, 1), inputs=[0]),                    # 1
        dict(conv_layer(rng, 16, 16, 3, 1, 1, resid=True), inputs=[1, 0]),     # 2 (+ residual 0)
        {"type": "maxpool", "inputs": [2], "params": dict(kh=2, kw=2, sh=2, sw=2, ph=0, pw=0)},
        dict(conv_layer(rng, 16, 16, 3, 1, 1, act="relu6", dw=True), inputs=[3]),
        dict(conv_layer(rng, 16, 32, 1, 1, 0), inputs=[4]),
        {"type": "gap", "inputs": [5]},
        {"type": "dense", "inputs": [6], "params": dict(in_features=32, out_features=10, act="none"),
         "weight": (0.3 * rng.standard_normal((10, 32))).astype(F32), "bias": np.zeros(10, F32)},
    ]


def test_whole_net_in_qint8_matches_oracle_bit_for_bit():
    import torch
    rng = np.random.default_rng(41)
    layers = small_net(rng)
    x = rng.standard_normal((2, 3, 16, 16)).astype(F32)
    s_in, scales = q8.calibrate(layers, x)
    g = build_graph(layers, x.shape, ("f32", "nchw"), ("f32", "nchw"), [("qi8", "nhwc")])
    g.set_qscale(-1, float(s_in))
    for i, s in enumerate(scales):
        g.set_qscale(i, float(s))
    used = _force(g, g.cost_table(), ["conv2/igemm_dp4a"])
    assert "conv2/igemm_dp4a" in used and "conv2/direct" in used
    y = g.run(to_device(x, ("f32", "nchw")))
    torch.cuda.synchronize()
    got = from_device(y, ("f32", "nchw"))
    want = q8.run_net_q8(layers, x, s_in, scales).astype(np.float64)
    assert np.array_equal(got.reshape(want.shape), want)
    # and within the quantisation budget of the float net
    ref = run_net(layers, x)
    assert maxrel(got.reshape(ref.shape), ref) < 0.1


def test_run_without_scales_is_a_state_error():
    rng = np.random.default_rng(43)
    layers = small_net(rng)[:2]
    g = build_graph(layers, (1, 3, 8, 8), ("f32", "nchw"), ("f32", "nchw"), [("qi8", "nhwc")])
    _force(g, g.cost_table(), [])
    from paper_2110_06037_gb300 import SnError
    with pytest.raises(SnError) as e:
        g.run(to_device(np.zeros((1, 3, 8, 8), F32), ("f32", "nchw")))
    assert "SN_ESTATE" in str(e.value)


def test_calibration_matches_the_float_oracle():
    import torch
    rng = np.random.default_rng(44)
    layers = small_net(rng)
    x = rng.standard_normal((2, 3, 16, 16)).astype(F32)
    g = build_graph(layers, x.shape, ("f32", "nchw"), ("f32", "nchw"), [("f32", "nhwc"), ("qi8", "nhwc")])
    g.profile(warmup=1, iters=3, topk=0)
    g.calibrate(to_device(x, ("f32", "nchw")))
    torch.cuda.synchronize()
    s_in, scales = q8.calibrate(layers, x)
    assert abs(g.get_qscale(-1) - s_in) <= 1e-6 * s_in
    for i, s in enumerate(scales):
        assert abs(g.get_qscale(i) - s) <= 1e-3 * s, i


def test_hybrid_dprs_equals_brute_force_and_runs():
    import torch
    rng = np.random.default_rng(45)
    layers = small_net(rng)
    x = rng.standard_normal((2, 3, 16, 16)).astype(F32)
    schemas = [("f16", "nhwc"), ("qi8", "nhwc")]
    g = build_graph(layers, x.shape, ("f32", "nchw"), ("f32", "nchw"), schemas)
    g.profile(warmup=1, iters=3, topk=1, passes=2)
    g.calibrate(to_device(x, ("f32", "nchw")))
    brute, _, _ = g.select_path(method=1)
    dprs, sch, _ = g.select_path()
    assert dprs == brute < 2**62
    y = g.run(to_device(x, ("f32", "nchw")))
    torch.cuda.synchronize()
    ref = run_net(layers, x)
    got = from_device(y, ("f32", "nchw"))
    assert maxrel(got.reshape(ref.shape), ref) < 0.1


# ------------------------------------------------------- fused boundaries
FUSED_CASES = [
    ("conv2/direct", lambda rng: conv_layer(rng, 8, 12, 3, 1, 1, act="relu6")),
    ("conv2/igemm_dp4a", lambda rng: conv_layer(rng, 16, 20, 3, 2, 1)),
    ("dwconv2/direct", lambda rng: conv_layer(rng, 16, 16, 3, 1, 1, dw=True)),
    ("maxpool/direct", lambda rng: {"type": "maxpool", "inputs": [-1],
                                    "params": dict(kh=3, kw=3, sh=2, sw=2, ph=1, pw=1)}),
    ("gap/reduce", lambda rng: {"type": "gap", "inputs": [-1]}),
    ("add/eltwise", lambda rng: {"type": "add", "inputs": [-1, -1], "params": dict(act="relu")}),
]


@pytest.mark.parametrize("out_dt", ["f16", "f32", "bf16"])
@pytest.mark.parametrize("case", range(len(FUSED_CASES)))
def test_fused_dequantisation_matches_oracle(case, out_dt):
    """A qint8 routine writing a float schema: the fp32 result rounded to that
    dtype, bit for bit."""
    import torch
    name, make = FUSED_CASES[case]
    rng = np.random.default_rng(500 + case)
    layer = make(rng)
    c = layer["params"]["c_in"] if "c_in" in layer.get("params", {}) else 16
    q_in = rng.integers(-127, 128, (2, c, 11, 9)).astype(np.int8)
    s_in = F32(0.04)
    scales = _out_scales([layer], q_in, s_in)
    sch = [("qi8", "nhwc"), (out_dt, "nhwc")]
    g = build_graph([layer], q_in.shape, ("qi8", "nhwc"), (out_dt, "nhwc"), sch)
    g.set_qscale(-1, float(s_in))
    g.set_qscale(0, float(scales[0]))
    t = g.cost_table()
    hit = [k for k in range(len(t["cost"])) if t["layer"][k] == 1 and routine_name(int(t["routine"][k])) == name
           and t["schema"][k] == 0 and t["out_schema"][k] == 1]
    assert hit, name
    g.set_path([int(np.flatnonzero(t["layer"] == 0)[0]), hit[0], int(np.flatnonzero(t["layer"] == 2)[0])])
    y = g.run(codes_to_device(q_in, "nhwc"))
    torch.cuda.synchronize()
    got = from_device(y, (out_dt, "nhwc"))
    n_in = len(layer["inputs"])
    want = q8.run_layer(layer, [q_in] * n_in, [s_in] * n_in, scales[0], out_dtype=out_dt).astype(np.float64)
    assert np.array_equal(got.reshape(want.shape), want), name
    # one launch: no dequantise adapt on the path
    assert g.plan_stats()[0] == 1


def test_hybrid_with_fused_boundaries_equals_exhaustive_search_and_runs():
    import torch
    from oracle.paths import brute_force_candidates
    rng = np.random.default_rng(46)
    layers = small_net(rng)[:5]  # stem, conv, residual conv, pool, depthwise
    x = rng.standard_normal((1, 3, 16, 16)).astype(F32)
    g = build_graph(layers, x.shape, ("f16", "nhwc"), ("f16", "nhwc"), [("f16", "nhwc"), ("qi8", "nhwc")])
    g.profile(warmup=1, iters=3, topk=1, passes=2)
    g.calibrate(to_device(x, ("f16", "nhwc")))
    t = g.cost_table()
    assert (t["out_schema"] != t["schema"]).any()
    per = []  # per layer the fastest candidate of each (read, written) pair (Eq. 1)
    for i in range(t["n_layers"]):
        best = {}
        for c in np.flatnonzero(t["layer"] == i):
            key = (int(t["schema"][c]), int(t["out_schema"][c]))
            if key not in best or t["cost"][c] < best[key]:
                best[key] = int(t["cost"][c])
        per.append([(v, k[0], k[1]) for k, v in sorted(best.items())])
    ref, _ = brute_force_candidates(per, t["edges"].tolist(), t["adapt"])
    tot, _, _ = g.select_path()
    assert tot == ref
    y = g.run(to_device(x, ("f16", "nhwc")))
    torch.cuda.synchronize()
    want = run_net(layers, x)
    assert maxrel(from_device(y, ("f16", "nhwc")).reshape(want.shape), want) < 0.1
