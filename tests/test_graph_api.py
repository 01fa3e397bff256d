"""Host-side behaviour of the C ABI: validation, call order, cost-table and
plan-file round trips.  CPU only (no kernel is launched)."""
import numpy as np
import pytest

import synth
from paper_2110_06037_gb300 import SN_SELECT_DPRS, SnError, build_graph, _sn
from paper_2110_06037_gb300.api import Graph

S2 = [("f32", "nchw"), ("f32", "nhwc")]


def tiny():
    x, layers = synth.tiny_cnn()
    return x, build_graph(layers, x.shape, ("f32", "nchw"), ("f32", "nchw"), S2, torch_alloc=False)


def test_shapes_and_candidates():
    x, g = tiny()
    t = g.cost_table()
    assert t["n_layers"] == 8 and t["n_schemas"] == 2
    assert g.layer_shape(1) == (1, 16, 32, 32)
    assert g.layer_shape(2) == (1, 32, 16, 16)
    assert g.layer_shape(6) == (1, 10, 1, 1)
    assert g.layer_shape(7) == (1, 10, 1, 1)
    # Winograd only on the 3x3 stride-1 conv, tensor cores never in fp32
    names = {(int(t["layer"][c]), _sn.routine_name(int(t["routine"][c]))) for c in range(len(t["cost"]))}
    assert (1, "conv2/wino_f2x2_3x3") in names and (2, "conv2/wino_f2x2_3x3") not in names
    assert not any(n == "conv2/igemm_tc" for _, n in names)
    assert np.all(t["cost"][t["routine"] != 0] == _sn.COST_INF)


def test_invalid_layers_rejected():
    g = Graph((1, 3, 8, 8), ("f32", "nchw"), ("f32", "nchw"), S2, torch_alloc=False)
    bad = dict(c_in=4, c_out=8, kh=3, kw=3, sh=1, sw=1, ph=1, pw=1)
    with pytest.raises(SnError) as e:
        g.add_layer(_sn.SN_L_CONV2, bad, (-1,), np.zeros((8, 4, 3, 3)), None)
    assert e.value.status == _sn.SN_EINVAL
    with pytest.raises(SnError):
        g.add_layer(_sn.SN_L_CONV2, dict(bad, c_in=3), (5,), np.zeros((8, 3, 3, 3)), None)
    with pytest.raises(SnError):
        g.add_layer(_sn.SN_L_CONV2, dict(bad, c_in=3, kh=11, ph=0), (-1,), np.zeros((8, 3, 11, 3)), None)
    with pytest.raises(SnError):
        g.add_layer(_sn.SN_L_DENSE, dict(in_features=3, out_features=2), (-1,), np.zeros((2, 3)), None)
    l0 = g.add_layer(_sn.SN_L_CONV2, dict(bad, c_in=3), (-1,), np.zeros((8, 3, 3, 3)), None)
    with pytest.raises(SnError):  # shapes differ
        g.add_layer(_sn.SN_L_ADD, {"act": "none"}, (-1, l0))


def test_dead_end_layer_is_rejected():
    g = Graph((1, 4, 4, 4), ("f32", "nchw"), ("f32", "nchw"), S2, torch_alloc=False)
    p = dict(c_in=4, c_out=4, kh=1, kw=1, sh=1, sw=1, ph=0, pw=0)
    g.add_layer(_sn.SN_L_CONV2, p, (-1,), np.zeros((4, 4, 1, 1)), None)
    g.add_layer(_sn.SN_L_CONV2, p, (-1,), np.zeros((4, 4, 1, 1)), None)  # layer 0 is now a dead end
    with pytest.raises(SnError) as e:
        g.cost_table()
    assert e.value.status == _sn.SN_EINVAL


def test_call_order():
    x, g = tiny()
    with pytest.raises(SnError) as e:
        _sn.check(_sn.lib().sn_run(g.h, 1, 1, None))
    assert e.value.status == _sn.SN_ESTATE
    with pytest.raises(SnError) as e:  # all costs unknown -> infeasible
        g.select_path(SN_SELECT_DPRS)
    assert e.value.status == _sn.SN_EINFEASIBLE
    with pytest.raises(SnError) as e:  # finalised: no more layers
        g.add_layer(_sn.SN_L_GAP, None, (0,))
    assert e.value.status == _sn.SN_ESTATE


def test_cost_table_validation_and_roundtrip(tmp_path):
    x, g = tiny()
    t = g.cost_table()
    rng = np.random.default_rng(0)
    t["cost"] = np.where(t["routine"] == 0, 0, rng.integers(1, 100, len(t["cost"]))).astype(np.int64)
    a = rng.integers(1, 50, t["adapt"].shape).astype(np.int64)
    for e in range(a.shape[0]):
        np.fill_diagonal(a[e], 0)
    t["adapt"] = a
    g.set_cost_table(t)
    t2 = g.cost_table()
    assert np.array_equal(t2["cost"], t["cost"]) and np.array_equal(t2["adapt"], a)
    bad = dict(t)
    bad["adapt"] = a.copy()
    bad["adapt"][0, 0, 0] = 5  # void adapt must be 0
    with pytest.raises(SnError):
        g.set_cost_table(bad)
    bad = dict(t)
    bad["schema"] = t["schema"].copy()
    bad["schema"][3] ^= 1
    with pytest.raises(SnError):
        g.set_cost_table(bad)
    assert np.array_equal(g.cost_table()["cost"], t["cost"])  # unchanged after errors
    tot, sch, cand = g.select_path(SN_SELECT_DPRS)
    p = tmp_path / "plan.json"
    g.save_plan(p)
    x2, g2 = tiny()
    g2.load_plan(p)
    t3 = g2.cost_table()
    assert np.array_equal(t3["cost"], t["cost"]) and np.array_equal(t3["adapt"], a)
    g2.save_plan(tmp_path / "plan2.json")
    assert open(p).read() == open(tmp_path / "plan2.json").read()


def test_set_path_validation():
    x, g = tiny()
    t = g.cost_table()
    with pytest.raises(SnError):
        g.set_path(np.zeros(t["n_layers"], np.int32))  # candidate 0 belongs to layer 0 only
    first = [int(np.flatnonzero(t["layer"] == i)[0]) for i in range(t["n_layers"])]
    g.set_path(first)


def test_tc_not_offered_where_it_cannot_run():
    for C, dt, lay, s, H in [(3, "f16", "nhwc", 1, 8), (64, "f32", "nhwc", 1, 8), (64, "f16", "nchw", 1, 8),
                             (64, "bf16", "nhwc", 2, 7)]:
        layer = synth.conv(C, 64, 3, s, 1)
        layer["weight"] = np.zeros((64, C, 3, 3), np.float32)
        layer["bias"] = np.zeros(64, np.float32)
        g = build_graph([dict(layer, inputs=[-1])], (1, C, H, H), (dt, lay), (dt, lay), [(dt, lay)],
                        torch_alloc=False)
        t = g.cost_table()
        assert not any(_sn.routine_name(int(r)) == "conv2/igemm_tc" for r in t["routine"])


def test_qint8_candidates_and_scales():
    """The qint8 schema offers exactly the routines with an int8 kernel, and
    blob scales are validated and kept across finalisation."""
    x, layers = synth.tiny_cnn()
    g = build_graph(layers, x.shape, ("f32", "nchw"), ("f32", "nchw"), [("f32", "nhwc"), ("qi8", "nhwc")],
                    torch_alloc=False)
    g.set_qscale(-1, 0.5)
    t = g.cost_table()  # finalises
    q8_names = {_sn.routine_name(int(t["routine"][c])) for c in range(len(t["cost"]))
                if t["schema"][c] == 1}
    assert q8_names <= {"io", "conv2/direct", "conv2/igemm_dp4a", "dwconv2/direct", "maxpool/direct", "gap/reduce",
                        "add/eltwise", "mul/eltwise", "dense/simt"}
    assert "conv2/direct" in q8_names
    f_names = {_sn.routine_name(int(t["routine"][c])) for c in range(len(t["cost"])) if t["schema"][c] == 0}
    assert "conv2/igemm_dp4a" not in f_names
    assert g.get_qscale(-1) == 0.5 and g.get_qscale(0) == 0.0
    g.set_qscale(2, 0.125)
    assert g.get_qscale(2) == 0.125
    for bad in (0.0, -1.0, float("inf"), float("nan")):
        with pytest.raises(SnError) as e:
            g.set_qscale(0, bad)
        assert e.value.status == _sn.SN_EINVAL
    with pytest.raises(SnError):
        g.set_qscale(len(layers), 1.0)
    with pytest.raises(SnError):
        g.get_qscale(-2)


def test_convert_needs_a_scale_for_qint8():
    import ctypes as C
    shp = (C.c_int64 * 4)(1, 2, 3, 4)
    fake = C.c_void_p(256)  # validation fails before any device access
    st = _sn.lib().sn_convert(fake, _sn.schema(("f16", "nchw")), fake, _sn.schema(("qi8", "nchw")), shp, None)
    assert st == _sn.SN_EINVAL
    st = _sn.lib().sn_convert_q(fake, _sn.schema(("f16", "nchw")), fake, _sn.schema(("f16", "nhwc")), shp,
                                C.c_float(1.0), None)
    assert st == _sn.SN_EINVAL  # no qint8 side
    st = _sn.lib().sn_convert_q(fake, _sn.schema(("f16", "nchw")), fake, _sn.schema(("qi8", "nchw")), shp,
                                C.c_float(0.0), None)
    assert st == _sn.SN_EINVAL  # bad scale


def test_calibration_needs_costs_and_a_single_input():
    import ctypes as C
    x, layers = synth.tiny_cnn()
    g = build_graph(layers, x.shape, ("f32", "nchw"), ("f32", "nchw"), [("f32", "nhwc"), ("qi8", "nhwc")],
                    torch_alloc=False)
    fake = C.c_void_p(256)  # refused before any device access
    assert _sn.lib().sn_calibrate(g.h, fake, None) == _sn.SN_ESTATE  # nothing profiled: no finite float path
    g2 = Graph((1, 4, 3, 3), ("f32", "nchw"), ("f32", "nchw"), [("f32", "nchw")], torch_alloc=False)
    g2.add_input((1, 4, 3, 3))
    w = np.zeros((4, 4, 1, 1), np.float32)
    p = dict(c_in=4, c_out=4, kh=1, kw=1, sh=1, sw=1, ph=0, pw=0)
    g2.add_layer(_sn.SN_L_CONV2, p, (-1,), w, None)
    g2.add_layer(_sn.SN_L_CONV2, p, (-2,), w, None)
    g2.add_layer(_sn.SN_L_ADD, dict(act="none"), (0, 1), None, None)
    assert _sn.lib().sn_calibrate(g2.h, fake, None) == _sn.SN_EUNSUPPORTED
    assert g2.io_counts() == (2, 1)
    # a second input's scale is set by its id
    g2.set_qscale(-2, 0.25)
    assert g2.get_qscale(-2) == 0.25 and g2.get_qscale(-1) == 0.0
    with pytest.raises(SnError):
        g2.set_qscale(-3, 1.0)


def test_candidate_descriptors():
    """Every candidate has a descriptor naming its routine, the schema it reads
    and, for the tensor-core routine, the parameter values that tell its
    variants apart (section III-C: routine descriptor + routine parameters)."""
    x, layers = synth.single_conv(2, 14, 64, 128, 3, 1)
    g = build_graph(layers, x.shape, ("bf16", "nhwc"), ("bf16", "nhwc"), [("bf16", "nhwc")], torch_alloc=False)
    t = g.cost_table()
    descs = [g.candidate_desc(c) for c in range(len(t["cost"]))]
    for c, d in enumerate(descs):
        assert d.startswith(_sn.routine_name(int(t["routine"][c]))), d
        assert "bf16.nhwc" in d or t["routine"][c] == 0, d
    tc = [d for c, d in enumerate(descs) if _sn.routine_name(int(t["routine"][c])) == "conv2/igemm_tc"]
    assert len(tc) > 4 and len(set(tc)) == len(tc), tc  # distinct parameter values per variant
    assert all("bn=" in d and "tile=" in d for d in tc)
    with pytest.raises(SnError):
        g.candidate_desc(len(t["cost"]))
