"""Seeded synthetic inputs and nets shaped like the paper's workloads.

This module holds random numbers and layer shapes only -- none of the
method's arithmetic.  It is the one piece both the CUDA path's tests and the
oracle consume: the tests draw arrays here and hand the same arrays to each.

Recipe (one numpy default_rng(seed) stream per net): the input is drawn first,
then every layer's weight in layer order, then every layer's bias in layer
order.  Weights are He-normal, N(0, 2/fan_in) with fan_in = C/groups * R * S
(variance 2/fan_in).  Biases stand for batch norm folded into the conv
(section III-A); they are N(0, 0.01) read as variance 0.01 (std 0.1).

The paper's trained VGG16/ResNet50/MobileNetV2/V3 weights and their datasets
are not available; these seeded tensors of the same architectures stand in.

Layer dicts follow the plain-data net description used by the tests:
    {"name", "type", "inputs", "params", "weight", "bias"}
type in conv2 | dwconv2 | maxpool | gap | add | dense; inputs are earlier
layer indices (-1 = net input); the last layer is the net output.
"""
from __future__ import annotations

import numpy as np


def conv(c_in, c_out, k, s=1, p=None, act="relu", groups=1, d=1, name=""):
    if p is None:
        p = (k // 2) * d
    return {"name": name, "type": "conv2" if groups == 1 or groups != c_in else "dwconv2",
            "params": dict(c_in=c_in, c_out=c_out, kh=k, kw=k, sh=s, sw=s, ph=p, pw=p,
                           dh=d, dw=d, groups=groups, act=act)}


def dwconv(c, k=3, s=1, act="relu6", name=""):
    p = k // 2
    return {"name": name, "type": "dwconv2",
            "params": dict(c_in=c, c_out=c, kh=k, kw=k, sh=s, sw=s, ph=p, pw=p, dh=1, dw=1,
                           groups=c, act=act)}


def maxpool(k=3, s=2, p=1, name=""):
    return {"name": name, "type": "maxpool", "params": dict(kh=k, kw=k, sh=s, sw=s, ph=p, pw=p)}


def gap(name=""):
    return {"name": name, "type": "gap", "params": {}}


def add(act="none", name=""):
    return {"name": name, "type": "add", "params": dict(act=act)}


def mul(act="none", name=""):
    """Per-channel scale: inputs (blob, N x C x 1 x 1 scale)."""
    return {"name": name, "type": "mul", "params": dict(act=act)}


def dense(fin, fout, act="none", name=""):
    return {"name": name, "type": "dense", "params": dict(in_features=fin, out_features=fout,
                                                          act=act)}


class _Builder:
    def __init__(self):
        self.layers = []

    def push(self, layer, inputs):
        layer = dict(layer)
        layer["inputs"] = list(inputs)
        self.layers.append(layer)
        return len(self.layers) - 1


def _weight_shape(layer):
    p = layer["params"]
    if layer["type"] in ("conv2", "dwconv2"):
        g = p["groups"]
        return (p["c_out"], p["c_in"] // g, p["kh"], p["kw"])
    if layer["type"] == "dense":
        return (p["out_features"], p["in_features"])
    return None


def _bias_len(layer):
    p = layer["params"]
    if layer["type"] in ("conv2", "dwconv2"):
        return p["c_out"]
    if layer["type"] == "dense":
        return p["out_features"]
    return None


def materialise(layers, input_shape, seed=0, input_dist="normal", weight_gain=None):
    """Draw the input, then weights in layer order, then biases, from one rng.

    input_dist: 'normal' = N(0,1), 'uniform' = U[-1, 1].
    weight_gain: optional {layer index: factor} applied to He-normal weights
    (used for the folded-BN scale of residual branches, see resnet50()).
    Returns (x float32 NCHW, layers with 'weight' and 'bias' filled in).
    """
    rng = np.random.default_rng(seed)
    if input_dist == "normal":
        x = rng.standard_normal(input_shape, dtype=np.float64).astype(np.float32)
    else:
        x = rng.uniform(-1.0, 1.0, size=input_shape).astype(np.float32)
    out = [dict(l) for l in layers]
    for i, l in enumerate(out):
        shp = _weight_shape(l)
        if shp is None:
            continue
        fan_in = int(np.prod(shp[1:]))
        w = rng.standard_normal(shp, dtype=np.float64) * np.sqrt(2.0 / fan_in)
        if weight_gain and i in weight_gain:
            w = w * weight_gain[i]
        l["weight"] = w.astype(np.float32)
    for l in out:
        n = _bias_len(l)
        if n is None:
            continue
        l["bias"] = (rng.standard_normal(n, dtype=np.float64) * 0.1).astype(np.float32)
    return x, out


# ----------------------------------------------------------------------------
# nets
# ----------------------------------------------------------------------------

def tiny_cnn(seed=0):
    """1x3x32x32 U[-1,1]; conv3x3 3->16 s1 + ReLU; conv3x3 16->32 s2 + ReLU;
    depthwise 3x3 32ch s1 + ReLU; conv1x1 32->64 + ReLU; GAP; FC 64->10."""
    b = _Builder()
    l = b.push(conv(3, 16, 3, 1, act="relu", name="conv1"), [-1])
    l = b.push(conv(16, 32, 3, 2, act="relu", name="conv2"), [l])
    l = b.push(dwconv(32, 3, 1, act="relu", name="dw3"), [l])
    l = b.push(conv(32, 64, 1, 1, act="relu", name="pw4"), [l])
    l = b.push(gap(name="gap"), [l])
    b.push(dense(64, 10, name="fc"), [l])
    return materialise(b.layers, (1, 3, 32, 32), seed, input_dist="uniform")


def mobilenet_v2(batch=1, seed=0, res=224):
    """MobileNetV2, width 1.0, ReLU6, BN folded; inverted residual blocks."""
    b = _Builder()
    l = b.push(conv(3, 32, 3, 2, act="relu6", name="stem"), [-1])
    c_in = 32
    cfg = [(1, 16, 1, 1), (6, 24, 2, 2), (6, 32, 3, 2), (6, 64, 4, 2), (6, 96, 3, 1),
           (6, 160, 3, 2), (6, 320, 1, 1)]
    blk = 0
    for t, c, n, s in cfg:
        for i in range(n):
            stride = s if i == 0 else 1
            hid = c_in * t
            x_in = l
            if t != 1:
                l = b.push(conv(c_in, hid, 1, 1, act="relu6", name=f"b{blk}.expand"), [l])
            l = b.push(dwconv(hid, 3, stride, act="relu6", name=f"b{blk}.dw"), [l])
            l = b.push(conv(hid, c, 1, 1, act="none", name=f"b{blk}.project"), [l])
            if stride == 1 and c_in == c:
                l = b.push(add(name=f"b{blk}.add"), [x_in, l])
            c_in = c
            blk += 1
    l = b.push(conv(c_in, 1280, 1, 1, act="relu6", name="head"), [l])
    l = b.push(gap(name="gap"), [l])
    b.push(dense(1280, 1000, name="fc"), [l])
    return materialise(b.layers, (batch, 3, res, res), seed)


def _make_divisible(v, d=8):
    """Round v to the nearest multiple of d, not below 90 % of v (MobileNet rule)."""
    r = max(d, int(v + d / 2) // d * d)
    return r + d if r < 0.9 * v else r


def mobilenet_v3(batch=1, seed=0, res=224):
    """MobileNetV3-Large, width 1.0, BN folded: hard-swish stem; fifteen
    bottlenecks (kernel, expansion, output, squeeze-excite, activation,
    stride); a 1x1 conv to 960 channels; GAP; a 960 -> 1280 hard-swish layer
    (the 1x1 conv on the pooled map, i.e. dense) and the 1280 -> 1000
    classifier.  Squeeze-excite: GAP -> dense to make_divisible(exp/4) + ReLU
    -> dense back to exp + hard sigmoid -> per-channel scale of the depthwise
    output."""
    spec = [(3, 16, 16, False, "relu", 1), (3, 64, 24, False, "relu", 2), (3, 72, 24, False, "relu", 1),
            (5, 72, 40, True, "relu", 2), (5, 120, 40, True, "relu", 1), (5, 120, 40, True, "relu", 1),
            (3, 240, 80, False, "hswish", 2), (3, 200, 80, False, "hswish", 1),
            (3, 184, 80, False, "hswish", 1), (3, 184, 80, False, "hswish", 1),
            (3, 480, 112, True, "hswish", 1), (3, 672, 112, True, "hswish", 1),
            (5, 672, 160, True, "hswish", 2), (5, 960, 160, True, "hswish", 1),
            (5, 960, 160, True, "hswish", 1)]
    b = _Builder()
    l = b.push(conv(3, 16, 3, 2, act="hswish", name="stem"), [-1])
    c_in = 16
    for blk, (k, exp, out, se, nl, s) in enumerate(spec):
        x_in = l
        if exp != c_in:
            l = b.push(conv(c_in, exp, 1, 1, act=nl, name=f"b{blk}.expand"), [l])
        l = b.push(dwconv(exp, k, s, act=nl, name=f"b{blk}.dw"), [l])
        if se:
            red = _make_divisible(exp // 4)
            g = b.push(gap(name=f"b{blk}.se.gap"), [l])
            g = b.push(dense(exp, red, act="relu", name=f"b{blk}.se.fc1"), [g])
            g = b.push(dense(red, exp, act="hsigmoid", name=f"b{blk}.se.fc2"), [g])
            l = b.push(mul(name=f"b{blk}.se.scale"), [l, g])
        l = b.push(conv(exp, out, 1, 1, act="none", name=f"b{blk}.project"), [l])
        if s == 1 and c_in == out:
            l = b.push(add(name=f"b{blk}.add"), [x_in, l])
        c_in = out
    l = b.push(conv(c_in, 960, 1, 1, act="hswish", name="head"), [l])
    l = b.push(gap(name="gap"), [l])
    l = b.push(dense(960, 1280, act="hswish", name="fc1"), [l])
    b.push(dense(1280, 1000, name="fc2"), [l])
    return materialise(b.layers, (batch, 3, res, res), seed)


RESIDUAL_GAIN = 0.25


def resnet50(batch=1, seed=0, res=224):
    """ResNet-50 v1.5 (stride on the 3x3), blocks 3-4-6-3, BN folded.

    The folded-BN scale of the last conv of every residual branch is
    RESIDUAL_GAIN (the other folded scales are 1).  With unit scales the
    residual sums of a random-weight ResNet grow ~3x in variance per block and
    overflow fp16 by the last stage; a small last-BN scale is the usual
    remedy and keeps every activation well inside fp16 range.
    """
    b = _Builder()
    gains = {}
    l = b.push(conv(3, 64, 7, 2, 3, act="relu", name="stem"), [-1])
    l = b.push(maxpool(3, 2, 1, name="maxpool"), [l])
    c_in = 64
    for si, (mid, out, n, s) in enumerate([(64, 256, 3, 1), (128, 512, 4, 2),
                                            (256, 1024, 6, 2), (512, 2048, 3, 2)]):
        for i in range(n):
            stride = s if i == 0 else 1
            x_in = l
            t = b.push(conv(c_in, mid, 1, 1, act="relu", name=f"s{si}b{i}.c1"), [x_in])
            t = b.push(conv(mid, mid, 3, stride, act="relu", name=f"s{si}b{i}.c2"), [t])
            t = b.push(conv(mid, out, 1, 1, act="none", name=f"s{si}b{i}.c3"), [t])
            gains[t] = RESIDUAL_GAIN
            if i == 0:
                sc = b.push(conv(c_in, out, 1, stride, 0, act="none", name=f"s{si}b{i}.proj"),
                            [x_in])
            else:
                sc = x_in
            l = b.push(add(act="relu", name=f"s{si}b{i}.add"), [sc, t])
            c_in = out
    l = b.push(gap(name="gap"), [l])
    b.push(dense(2048, 1000, name="fc"), [l])
    return materialise(b.layers, (batch, 3, res, res), seed, weight_gain=gains)


def vgg16(batch=1, seed=0, res=224):
    """VGG16 (configuration D): thirteen 3x3 convs with ReLU in five groups,
    each followed by a 2x2 stride-2 max pool, then three fully connected
    layers.  The first of them runs as a convolution whose kernel covers the
    whole final feature map (res/32 square, valid padding): it is the dense
    layer over the flattened map, independent of the activation layout.
    He-normal weights keep the ReLU activations' variance level without BN.
    """
    if res % 32:
        raise ValueError("vgg16: the input side must be a multiple of 32")
    b = _Builder()
    l, c = -1, 3
    groups = [(64, 2), (128, 2), (256, 3), (512, 3), (512, 3)]
    for gi, (width, n) in enumerate(groups):
        for i in range(n):
            l = b.push(conv(c, width, 3, 1, 1, act="relu", name=f"conv{gi + 1}_{i + 1}"), [l])
            c = width
        l = b.push(maxpool(2, 2, 0, name=f"pool{gi + 1}"), [l])
    f = res // 32
    l = b.push(conv(512, 4096, f, 1, 0, act="relu", name="fc6"), [l])
    l = b.push(dense(4096, 4096, act="relu", name="fc7"), [l])
    b.push(dense(4096, 1000, name="fc8"), [l])
    return materialise(b.layers, (batch, 3, res, res), seed)


def single_conv(N, H, C, K, k, s, seed=0, act="relu"):
    """One conv layer of the single-layer sweep: NxCxHxH N(0,1), He-normal."""
    b = _Builder()
    b.push(conv(C, K, k, s, act=act, name=f"conv{k}x{k}s{s}"), [-1])
    return materialise(b.layers, (N, C, H, H), seed)


def random_dag(rng, n_inner, p_edge=0.35, max_in=3):
    """A random 1-in-1-out DAG over n_inner + 2 layers (0 = input, last = output).

    Every layer is reachable from the input and reaches the output.  Returns
    the edge list (src, dst) with src < dst.
    """
    n = n_inner + 2
    edges = set()
    for v in range(1, n - 1):
        preds = [u for u in range(0, v) if rng.random() < p_edge][:max_in]
        if not preds:
            preds = [int(rng.integers(0, v))]
        for u in preds:
            edges.add((u, v))
    has_succ = {u for u, _ in edges}
    for u in range(0, n - 1):
        if u not in has_succ:
            edges.add((u, n - 1) if u == 0 or rng.random() < 0.5 or u == n - 2
                      else (u, int(rng.integers(u + 1, n))))
    # make sure the output has a predecessor and every non-output layer has a successor
    changed = True
    while changed:
        changed = False
        has_succ = {u for u, _ in edges}
        for u in range(0, n - 1):
            if u not in has_succ:
                edges.add((u, n - 1))
                changed = True
    return sorted(edges)
