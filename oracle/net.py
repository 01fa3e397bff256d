"""Oracle forward pass of a whole net, layer by layer, in fp64.

TEST INFRASTRUCTURE ONLY (see the package docstring).

A net is the plain-data description used throughout the tests: a list of
layers in topological order (section IV-A numbers them L_1..L_n the same way),
each a dict with keys
    type    'conv2' | 'dwconv2' | 'maxpool' | 'gap' | 'add' | 'dense' | 'mul'
    inputs  list of earlier layer indices, -1 = the net input
    params  dict of layer parameters (section III-B)
    weight, bias   fp32 arrays (conv: [K, C/groups, R, S]; dense: [out, in])
The last layer is the net output.

Precision: for an fp16/bf16 schema the GPU stores the input and the weights
in that format, so the oracle takes them as stored (rounded to nearest even,
widened exactly) and then computes in fp64 with no intermediate rounding.
Biases are kept in fp32 by every routine, so they are used unrounded.
"""
from __future__ import annotations

import numpy as np

from . import add, conv2d, dense, gap, maxpool2d, mul, round_to


def run_layer(layer: dict, inputs: list, dtype: str = "f32") -> np.ndarray:
    """One layer on fp64 NCHW inputs; weights are taken as stored in `dtype`."""
    t, p = layer["type"], layer.get("params", {})
    if t in ("conv2", "dwconv2"):
        w = round_to(layer["weight"], dtype)
        b = layer.get("bias")
        groups = p.get("groups", 1) if t == "conv2" else p["c_in"]
        if len(inputs) == 2:
            # conv2 with a residual input: the activation applies to
            # conv + bias + residual, with no rounding in between
            y = conv2d(inputs[0], w, b, stride=(p["sh"], p["sw"]), pad=(p["ph"], p["pw"]),
                       dil=(p.get("dh", 1), p.get("dw", 1)), groups=groups, act="none")
            return add(y, inputs[1], act=p.get("act", "none"))
        return conv2d(inputs[0], w, b, stride=(p["sh"], p["sw"]), pad=(p["ph"], p["pw"]),
                      dil=(p.get("dh", 1), p.get("dw", 1)), groups=groups,
                      act=p.get("act", "none"))
    if t == "maxpool":
        return maxpool2d(inputs[0], k=(p["kh"], p["kw"]), stride=(p["sh"], p["sw"]),
                         pad=(p["ph"], p["pw"]))
    if t == "gap":
        return gap(inputs[0])
    if t == "add":
        return add(inputs[0], inputs[1], act=p.get("act", "none"))
    if t == "mul":
        return mul(inputs[0], inputs[1], act=p.get("act", "none"))
    if t == "dense":
        w = round_to(layer["weight"], dtype)
        return dense(inputs[0], w, layer.get("bias"), act=p.get("act", "none"))
    raise ValueError(f"unknown layer type {t}")


def run_net(layers: list, x, dtype: str = "f32", keep: bool = False):
    """Whole net from the input as stored in `dtype`.

    x is the net input, or a list of net inputs for ids -1, -2, ... (several
    input layers under the auxiliary input layer, section IV-E).  Returns the
    last layer's output (fp64 NCHW), or (output, [every layer's output]) when
    keep=True.
    """
    xs = list(x) if isinstance(x, (list, tuple)) else [x]
    x0s = [round_to(np.asarray(v, np.float32), dtype).astype(np.float64) for v in xs]
    outs = []
    for layer in layers:
        ins = [x0s[-1 - j] if j < 0 else outs[j] for j in layer["inputs"]]
        outs.append(run_layer(layer, ins, dtype))
    return (outs[-1], outs) if keep else outs[-1]
