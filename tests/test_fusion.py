"""The residual-add fusion pass and the conv2-with-residual layer, on the CPU.

  * fuse_residual folds every ResNet-50 / MobileNetV2 residual add into the
    conv2 that feeds it and leaves a valid topological net;
  * the oracle's fused layer equals conv2 followed by add exactly (fp64, the
    same operations in the same order), on a small residual net and on
    ResNet-50 at a small resolution;
  * a residual of the wrong shape is rejected; only the direct and the
    tensor-core routines are offered for a fused layer;
  * DPRS on the fused nets equals the oracle's block-wise exact search."""
import numpy as np
import pytest

import synth
from oracle.net import run_net
from paper_2110_06037_gb300 import SnError, _sn, build_graph, fuse_residual, fused_description
from paper_2110_06037_gb300.api import Graph

from test_dprs import check_against_oracle, random_costs


def _counts(layers):
    return (sum(1 for l in layers if l["type"] == "add"),
            sum(1 for l in layers if l["type"] == "conv2" and len(l["inputs"]) == 2))


def test_fuse_resnet50_and_mobilenet_v2_structure():
    xr, r50 = synth.resnet50(1, res=32)
    f = fuse_residual(r50, xr.shape)
    assert _counts(r50) == (16, 0) and _counts(f) == (0, 16)
    assert len(f) == len(r50) - 16
    xm, mb = synth.mobilenet_v2(1, res=32)
    fm = fuse_residual(mb, xm.shape)
    assert _counts(mb)[0] == 10 and _counts(fm) == (0, 10)
    for net in (f, fm):
        for i, l in enumerate(net):
            assert all(j < i for j in l["inputs"])  # topological
        used = {j for l in net for j in l["inputs"]}
        assert all(i in used for i in range(len(net) - 1))  # no dead ends
    # the fused layer takes the add's activation; a conv with an activation is left alone
    assert all(l["params"]["act"] == "relu" for l in f if len(l["inputs"]) == 2)
    x, tiny = synth.tiny_cnn()
    assert fuse_residual(tiny, x.shape) == tiny


def _residual_net(rng):
    """conv -> conv(act none) -> add(relu) with the first conv's output."""
    c1 = synth.conv(4, 6, 3, 1, 1, act="relu")
    c2 = synth.conv(6, 6, 3, 1, 1, act="none")
    for l in (c1, c2):
        k, c = l["params"]["c_out"], l["params"]["c_in"]
        l["weight"] = rng.standard_normal((k, c, 3, 3)).astype(np.float32)
        l["bias"] = rng.standard_normal(k).astype(np.float32)
    c1["inputs"], c2["inputs"] = [-1], [0]
    add = {"type": "add", "name": "add", "inputs": [1, 0], "params": {"act": "relu"}}
    gap = {"type": "gap", "name": "gap", "inputs": [2], "params": {}}
    return [c1, c2, add, gap]


def test_oracle_fused_equals_conv_then_add():
    rng = np.random.default_rng(3)
    net = _residual_net(rng)
    f = fuse_residual(net, (2, 4, 7, 5))
    assert [l["type"] for l in f] == ["conv2", "conv2", "gap"] and f[1]["inputs"] == [0, 0]
    x = rng.standard_normal((2, 4, 7, 5)).astype(np.float32)
    a = run_net(net, x, "f32")
    b = run_net(f, x, "f32")
    assert np.array_equal(a, b)


def test_oracle_fused_resnet50_equals_unfused():
    x, r50 = synth.resnet50(1, res=32)
    a = run_net(r50, x, "bf16")
    b = run_net(fuse_residual(r50, x.shape), x, "bf16")
    assert np.array_equal(a, b)


def test_residual_shape_checked_and_routines_offered():
    g = Graph((1, 8, 6, 6), ("f16", "nhwc"), ("f16", "nhwc"), [("f16", "nhwc"), ("f16", "nchw")],
              torch_alloc=False)
    p = dict(c_in=8, c_out=8, kh=3, kw=3, sh=1, sw=1, ph=1, pw=1)
    with pytest.raises(SnError) as e:  # stride 2 output is 3x3, the residual 6x6
        g.add_layer(_sn.SN_L_CONV2, dict(p, sh=2, sw=2), (-1, -1), np.zeros((8, 8, 3, 3), np.float32), None)
    assert e.value.status == _sn.SN_EINVAL
    with pytest.raises(SnError):  # depthwise takes one input
        g.add_layer(_sn.SN_L_DWCONV2, dict(p, groups=8), (-1, -1), np.zeros((8, 1, 3, 3), np.float32), None)
    g.add_layer(_sn.SN_L_CONV2, dict(p, act="relu"), (-1, -1), np.zeros((8, 8, 3, 3), np.float32), None)
    t = g.cost_table()
    names = {_sn.routine_name(int(t["routine"][c])) for c in range(len(t["cost"])) if t["layer"][c] == 1}
    assert names == {"conv2/direct", "conv2/igemm_tc"}


@pytest.mark.parametrize("net", ["resnet50", "mobilenet_v2"])
def test_dprs_on_fused_nets_equals_blockwise_search(net):
    _, layers = (synth.resnet50(1, res=32) if net == "resnet50" else synth.mobilenet_v2(1, res=32))
    layers = fuse_residual(layers, (1, 3, 32, 32))
    sch = [("f16", "nchw"), ("f16", "nhwc")]
    g = build_graph(layers, (1, 3, 32, 32), ("f32", "nchw"), ("f32", "nchw"), sch, torch_alloc=False)
    for seed in range(3):
        rng = np.random.default_rng(100 + seed)
        t = random_costs(g, rng, p_inf=0.05)
        check_against_oracle(g, t, exhaustive=False)


def test_library_pass_through_the_c_abi():
    """sn_fuse_residual on the graph itself (what a C caller gets): ResNet-50
    loses its 16 adds and 16 convs, the id map sends each add to its fused
    layer and each folded conv2 to -1, the outputs follow the map, and once
    the net is finalised the pass is refused with SN_ESTATE."""
    import ctypes as C
    x, r50 = synth.resnet50(1, res=32)
    g = build_graph(r50, x.shape, ("f16", "nchw"), ("f16", "nchw"), [("f16", "nhwc")], torch_alloc=False)
    m = len(r50)
    ids = (C.c_int32 * m)()
    nf = C.c_int32()
    assert _sn.lib().sn_fuse_residual(g.h, ids, m, C.byref(nf)) == _sn.SN_OK
    assert nf.value == 16
    new_id = list(ids)
    adds = [i for i, l in enumerate(r50) if l["type"] == "add"]
    assert sum(1 for v in new_id if v < 0) == 16
    assert all(new_id[i] >= 0 for i in adds)
    folded = [i for i, v in enumerate(new_id) if v < 0]
    assert all(r50[i]["type"] == "conv2" and r50[i]["params"]["act"] == "none" for i in folded)
    kept = [v for v in new_id if v >= 0]
    assert kept == list(range(m - 16))  # renumbered in order
    g.n_user = m - 16
    t = g.cost_table()
    assert t["n_layers"] == m - 16 + 2  # + the auxiliary input and output layers
    # one edge per layer input of the fused description, plus the output layer's
    assert len(t["edges"]) == sum(len(l["inputs"]) for l in fused_description(r50, new_id)) + 1
    with pytest.raises(SnError) as e:
        g.fuse_residual()
    assert e.value.status == _sn.SN_ESTATE


def test_library_pass_leaves_nets_without_residual_adds_alone():
    x, tiny = synth.tiny_cnn()
    g = build_graph(tiny, x.shape, ("f32", "nchw"), ("f32", "nchw"), [("f32", "nchw")], torch_alloc=False,
                    fuse=True)
    assert g.fused_ids == list(range(len(tiny)))
    # an add fed by a conv2 that has an activation, or by a conv2 read twice, stays
    rng = np.random.default_rng(5)
    net = _residual_net(rng)
    net[1]["params"] = dict(net[1]["params"], act="relu")
    g = build_graph(net, (2, 4, 7, 5), ("f32", "nchw"), ("f32", "nchw"), [("f32", "nchw")], torch_alloc=False,
                    fuse=True)
    assert g.fused_ids == [0, 1, 2, 3]
