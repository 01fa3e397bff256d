"""Build a Graph from the plain-data net description (list of layer dicts).

Each dict has 'type' (conv2 | dwconv2 | maxpool | gap | add | dense),
'inputs' (earlier layer indices, -1 = net input), 'params', and for conv and
dense layers 'weight' (fp32, conv [K][C/groups][R][S], dense [out][in]) and
'bias'.  Layer i of the list becomes layer id i of the graph.
"""
from __future__ import annotations

from . import _sn
from .api import Graph

TYPES = {"conv2": _sn.SN_L_CONV2, "dwconv2": _sn.SN_L_DWCONV2, "maxpool": _sn.SN_L_MAXPOOL,
         "gap": _sn.SN_L_GAP, "add": _sn.SN_L_ADD, "dense": _sn.SN_L_DENSE}


def build_graph(layers, in_shape, in_schema, out_schema, schemas, torch_alloc=True) -> Graph:
    g = Graph(in_shape, in_schema, out_schema, schemas, torch_alloc=torch_alloc)
    for i, l in enumerate(layers):
        lid = g.add_layer(TYPES[l["type"]], l.get("params"), tuple(l["inputs"]), l.get("weight"),
                          l.get("bias"))
        assert lid == i
    return g
