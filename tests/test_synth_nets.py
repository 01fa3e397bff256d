"""The synthetic workloads' structure (CPU): the layer sequences and output
shapes the builders promise, checked on the oracle at a small input side."""
import numpy as np

import synth
from oracle.net import run_net


def test_vgg16_structure_and_shapes():
    x, layers = synth.vgg16(2, res=64)
    kinds = [l["type"] for l in layers]
    assert kinds.count("conv2") == 14 and kinds.count("maxpool") == 5 and kinds.count("dense") == 2
    widths = [l["params"]["c_out"] for l in layers if l["type"] == "conv2"][:13]
    assert widths == [64, 64, 128, 128, 256, 256, 256, 512, 512, 512, 512, 512, 512]
    fc6 = [l for l in layers if l.get("name") == "fc6"][0]
    p = fc6["params"]
    assert (p["kh"], p["kw"], p["ph"], p["pw"], p["c_in"], p["c_out"]) == (2, 2, 0, 0, 512, 4096)
    for l in layers:
        if l["type"] == "maxpool":
            assert (l["params"]["kh"], l["params"]["sh"], l["params"]["ph"]) == (2, 2, 0)
    y = run_net(layers, x, "f32")
    assert y.shape == (2, 1000, 1, 1) and np.all(np.isfinite(y))


def test_vgg16_fc6_equals_dense_over_the_flattened_map():
    """The fc6 convolution (kernel = the whole final map, valid padding) is the
    dense layer over the map flattened in (c, h, w) order."""
    x, layers = synth.vgg16(1, res=64)
    i6 = [i for i, l in enumerate(layers) if l.get("name") == "fc6"][0]
    head = [dict(l) for l in layers[:i6]]
    feat = run_net(head, x, "f32").astype(np.float64)          # (1, 512, 2, 2)
    fc6 = layers[i6]
    w = fc6["weight"].astype(np.float64).reshape(4096, -1)      # [K, C*R*S] in (c, r, s) order
    ref = np.maximum(w @ feat.reshape(-1) + fc6["bias"], 0.0)
    got = run_net(layers[: i6 + 1], x, "f32").reshape(-1)
    assert np.max(np.abs(got - ref)) <= 1e-9 * max(1.0, np.max(np.abs(ref)))


def test_mobilenet_v3_large_structure():
    x, layers = synth.mobilenet_v3(1, res=64)
    kinds = [l["type"] for l in layers]
    assert kinds.count("dwconv2") == 15 and kinds.count("mul") == 8 and kinds.count("add") == 10
    dws = [l["params"]["kh"] for l in layers if l["type"] == "dwconv2"]
    assert dws == [3, 3, 3, 5, 5, 5, 3, 3, 3, 3, 3, 3, 5, 5, 5]
    # squeeze-excite widths: make_divisible(exp / 4, 8)
    red = [l["params"]["out_features"] for l in layers if l.get("name", "").endswith(".se.fc1")]
    assert red == [24, 32, 32, 120, 168, 168, 240, 240]
    acts = {l["params"].get("act") for l in layers if l["type"] in ("conv2", "dwconv2", "dense")}
    assert {"hswish", "hsigmoid", "relu", "none"} <= acts
    for l in layers:
        if l["type"] == "mul":
            assert layers[l["inputs"][1]].get("name", "").endswith(".se.fc2")
    y = run_net(layers, x, "f32")
    assert y.shape == (1, 1000, 1, 1) and np.all(np.isfinite(y))
