"""A net with two inputs and two outputs on the GPU (section IV-E):
profile -> DPRS -> run_multi, each output against the oracle, with and
without CUDA-graph replay; and a qint8 input scale given by its id."""
import numpy as np
import pytest

import oracle
import synth
from oracle.net import run_net
from paper_2110_06037_gb300 import SN_OPT_CUDA_GRAPH, SN_SELECT_BRUTE, SN_SELECT_DPRS, build_graph

from gpu_helpers import TOL, from_device, maxrel, to_device
from oracle.paths import blockwise_search
from test_dprs import has_fused, oracle_layer_cost, oracle_pair_cost

pytestmark = pytest.mark.gpu

F16 = [("f16", "nchw"), ("f16", "nhwc")]


def mimo_net(rng):
    """image (-1) -> stem conv -> block; side input (-2) -> 1x1 conv; sum ->
    head conv.  Outputs: the block (a feature map) and the head."""
    def conv(c, k, ks, s, inputs, act="relu"):
        l = synth.conv(c, k, ks, s, ks // 2, act=act)
        l["weight"] = (rng.standard_normal((k, c, ks, ks)) * np.sqrt(2.0 / (c * ks * ks))).astype(np.float32)
        l["bias"] = (0.1 * rng.standard_normal(k)).astype(np.float32)
        l["inputs"] = inputs
        return l
    return [
        conv(3, 32, 3, 2, [-1]),                               # 0
        conv(32, 32, 3, 1, [0]),                               # 1: output 0
        conv(16, 32, 1, 1, [-2], act="none"),                  # 2
        {"type": "add", "inputs": [1, 2], "params": {"act": "relu"}},  # 3
        conv(32, 64, 3, 2, [3]),                               # 4: output 1
    ]


def test_two_inputs_two_outputs_match_the_oracle():
    import torch
    rng = np.random.default_rng(77)
    layers = mimo_net(rng)
    x = rng.standard_normal((2, 3, 32, 32)).astype(np.float32)
    side = rng.standard_normal((2, 16, 16, 16)).astype(np.float32)
    g = build_graph(layers, x.shape, ("f16", "nchw"), ("f16", "nchw"), F16, extra_inputs=[side.shape],
                    outputs=[1, 4])
    assert g.io_counts() == (2, 2)
    g.profile(warmup=1, iters=5, topk=2, passes=3)
    t = g.cost_table()
    if has_fused(t):  # a routine that writes another schema: the exact pair-state search
        lcp, pairs = oracle_pair_cost(t)
        ref_cost, _ = blockwise_search(lcp, t["edges"], t["adapt"], pairs=pairs)
    else:
        ref_cost, _, _ = oracle.brute_force(oracle_layer_cost(t), t["edges"], t["adapt"])
    tot, _, _ = g.select_path(SN_SELECT_DPRS)
    assert tot == ref_cost
    assert g.select_path(SN_SELECT_BRUTE)[0] == tot
    g.select_path(SN_SELECT_DPRS)
    _, outs = run_net(layers, [x, side], "f16", keep=True)
    xs = [to_device(x, ("f16", "nchw")), to_device(side, ("f16", "nchw"))]
    for graph_mode in (0, 1):
        g.set_option(SN_OPT_CUDA_GRAPH, graph_mode)
        stream = torch.cuda.Stream()
        ys = g.run_multi(xs, stream=stream)
        stream.synchronize()
        assert len(ys) == 2
        for y, j in zip(ys, (1, 4)):
            got = from_device(y, ("f16", "nchw"))
            assert maxrel(got, outs[j]) <= TOL["f16"], (graph_mode, j)
    # the single-buffer call refuses a net with two inputs
    from paper_2110_06037_gb300 import SnError
    with pytest.raises(SnError):
        g.run(xs[0])
