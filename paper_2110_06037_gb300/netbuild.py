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
                outputs=None) -> Graph:
    """extra_inputs: shapes of net inputs -2, -3, ...; outputs: layer indices
    of the net outputs (default: the last layer)."""
    g = Graph(in_shape, in_schema, out_schema, schemas, torch_alloc=torch_alloc)
    for k, shp in enumerate(extra_inputs):
        assert g.add_input(shp) == -2 - k
    for i, l in enumerate(layers):
        lid = g.add_layer(TYPES[l["type"]], l.get("params"), tuple(l["inputs"]), l.get("weight"),
                          l.get("bias"))
        assert lid == i
    if outputs is not None:
        g.set_outputs(list(outputs))
    return g


def fuse_residual(layers):
    """Fuse every residual add into the convolution that feeds it.

    A graph-optimiser pass over the plain-data description, run before the
    net is built and tuned (the paper fuses layers ahead of tuning, section
    III-A): an 'add' whose input is a 'conv2' with no activation, read by
    nothing else, becomes that conv2 with the add's other input as a
    residual and the add's activation, y = act(conv(x) + b + residual).  The
    fused layer takes the add's place in the list (after both of its inputs)
    and the conv2 is dropped; indices are renumbered.  Returns a new list.
    """
    consumers = {}
    for i, l in enumerate(layers):
        for j in l["inputs"]:
            consumers.setdefault(j, []).append(i)
    fold = {}  # add index -> (conv index, residual index)
    for i, l in enumerate(layers):
        if l["type"] != "add":
            continue
        for pos in (0, 1):
            j, other = l["inputs"][pos], l["inputs"][1 - pos]
            if j < 0 or layers[j]["type"] != "conv2" or len(layers[j]["inputs"]) != 1:
                continue
            if layers[j]["params"].get("act", "none") != "none" or consumers.get(j) != [i]:
                continue
            fold[i] = (j, other)
            break
    dropped = {j for (j, _) in fold.values()}
    new_index, out = {}, []
    for i, l in enumerate(layers):
        if i in dropped:
            continue
        new_index[i] = len(out)
        if i in fold:
            j, other = fold[i]
            conv = layers[j]
            params = dict(conv["params"], act=l["params"].get("act", "none"))
            out.append(dict(conv, name=conv.get("name", "conv") + "+" + l.get("name", "add"), params=params,
                            inputs=[conv["inputs"][0], other]))
        else:
            out.append(dict(l))
    for l in out:
        l["inputs"] = [j if j < 0 else new_index[j] for j in l["inputs"]]
    return out
