"""Build a Graph from the plain-data net description (list of layer dicts).

Each dict has 'type' (conv2 | dwconv2 | maxpool | gap | add | dense),
'inputs' (earlier layer indices; -1, -2, ... = net inputs), 'params', and for conv and
dense layers 'weight' (fp32, conv [K][C/groups][R][S], dense [out][in]) and
'bias'.  Layer i of the list becomes layer id i of the graph.
"""
from __future__ import annotations

from . import _sn
from .api import Graph

TYPES = {"conv2": _sn.SN_L_CONV2, "dwconv2": _sn.SN_L_DWCONV2, "maxpool": _sn.SN_L_MAXPOOL,
         "gap": _sn.SN_L_GAP, "add": _sn.SN_L_ADD, "dense": _sn.SN_L_DENSE, "mul": _sn.SN_L_MUL}


def build_graph(layers, in_shape, in_schema, out_schema, schemas, torch_alloc=True, extra_inputs=(),
                outputs=None, fuse=False) -> Graph:
    """extra_inputs: shapes of net inputs -2, -3, ...; outputs: layer indices
    of the net outputs (default: the last layer).  fuse=True runs the
    library's residual-add fusion pass (sn_fuse_residual) before anything
    finalises the net; the graph then has the layers of
    fused_description(layers, g.fused_ids) and g.fused_ids maps the given
    layer indices to the graph's."""
    g = Graph(in_shape, in_schema, out_schema, schemas, torch_alloc=torch_alloc)
    for k, shp in enumerate(extra_inputs):
        assert g.add_input(shp) == -2 - k
    for i, l in enumerate(layers):
        lid = g.add_layer(TYPES[l["type"]], l.get("params"), tuple(l["inputs"]), l.get("weight"),
                          l.get("bias"))
        assert lid == i
    if outputs is not None:
        g.set_outputs(list(outputs))
    g.fused_ids = None
    if fuse:
        g.fused_ids, _ = g.fuse_residual()
    return g


def fused_description(layers, new_id):
    """The plain-data description of the net after the library's fusion pass,
    read off its id map (new_id[old], -1 for a folded conv2): a kept layer is
    copied with its inputs renumbered; an add one of whose inputs was folded
    becomes that conv2 with the add's other input as its residual and the
    add's activation.  This only restates, for the Python side, what
    sn_fuse_residual did to the graph."""
    out = [None] * (max(new_id) + 1 if new_id else 0)
    for i, l in enumerate(layers):
        k = new_id[i]
        if k < 0:
            continue
        folded = [j for j in l["inputs"] if j >= 0 and new_id[j] < 0] if l["type"] == "add" else []
        if folded:
            j = folded[0]
            other = l["inputs"][1] if l["inputs"][0] == j else l["inputs"][0]
            conv = layers[j]
            params = dict(conv["params"], act=l["params"].get("act", "none"))
            d = dict(conv, name=conv.get("name", "conv") + "+" + l.get("name", "add"), params=params,
                     inputs=[conv["inputs"][0], other])
        else:
            d = dict(l)
        d["inputs"] = [j if j < 0 else new_id[j] for j in d["inputs"]]
        out[k] = d
    return out


def fuse_residual(layers, in_shape, extra_inputs=(), outputs=None):
    """Run the library's residual-add fusion pass (sn_fuse_residual) on a
    host-only graph of the net and return the fused plain-data description
    (see fused_description)."""
    g = build_graph(layers, in_shape, ("f32", "nchw"), ("f32", "nchw"), [("f32", "nchw")], torch_alloc=False,
                    extra_inputs=extra_inputs, outputs=outputs, fuse=True)
    return fused_description(layers, g.fused_ids)
