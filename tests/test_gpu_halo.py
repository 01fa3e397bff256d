"""Halo-tile routine parameters of conv2/igemm_tc (3x3, stride 1).

A halo variant tiles the output in 8 x 16 pixels of one image; each K step is
one row of three taps of one 64-channel block, and its stage holds the 10 x 16
input pixels the row's three column taps read as a single TMA box, from which
the MMAs of the three taps start one box row apart.  On maps that are and are
not multiples of the tile, channel counts that are not multiples of 64 on
either side, padding 1 and 0, and a fused residual input:
  * every halo variant matches the oracle within the fp16/bf16 tolerance;
  * a second launch and a CUDA-graph replay give the same bits.
"""
import numpy as np
import pytest

import synth
from oracle.net import run_layer
from paper_2110_06037_gb300 import SN_OPT_CUDA_GRAPH, build_graph, routine_name

from gpu_helpers import TOL, from_device, maxrel, stored_values, to_device

pytestmark = pytest.mark.gpu

# (N, H, W, C, K, pad, residual, dtype)
CASES = [
    (2, 56, 56, 64, 64, 1, False, "bf16"),     # a ResNet-50 stage-1 layer at batch 2
    (2, 28, 28, 128, 128, 1, True, "f16"),     # stage 2, fused residual
    (3, 14, 14, 256, 256, 1, False, "bf16"),   # stage 3: tiles wider and taller than the map
    (2, 7, 7, 512, 512, 1, True, "bf16"),      # stage 4
    (2, 19, 23, 40, 72, 1, False, "f16"),      # ragged map, 40 -> 72 channels
    (1, 20, 18, 64, 128, 0, False, "bf16"),    # no padding: 18 x 16 output
]


def _graph(N, H, W, C, K, pad, res, dt, seed):
    rng = np.random.default_rng(seed)
    layer = synth.conv(C, K, 3, 1, pad, act="relu")
    layer["weight"] = (rng.standard_normal((K, C, 3, 3)) * np.sqrt(2.0 / (C * 9))).astype(np.float32)
    layer["bias"] = (rng.standard_normal(K) * 0.1).astype(np.float32)
    P, Q = H + 2 * pad - 2, W + 2 * pad - 2
    x = rng.standard_normal((N, C, H, W)).astype(np.float32)
    r = rng.standard_normal((N, K, P, Q)).astype(np.float32) if res else None
    sch = (dt, "nhwc")
    g = build_graph([dict(layer, inputs=[-1, -2] if res else [-1])], x.shape, sch, sch, [sch],
                    extra_inputs=[(N, K, P, Q)] if res else ())
    return g, layer, x, r, sch


@pytest.mark.parametrize("case", CASES, ids=lambda c: "n%d_%dx%d_%d-%d_p%d%s_%s" % (
    c[0], c[1], c[2], c[3], c[4], c[5], "_res" if c[6] else "", c[7]))
def test_halo_variants_match_oracle_and_repeat_bit_for_bit(case):
    import torch
    N, H, W, C, K, pad, res, dt = case
    g, layer, x, r, sch = _graph(*case, seed=N * 1000 + H * 10 + C + K)
    t = g.cost_table()
    io = [int(np.flatnonzero(t["layer"] == i)[0]) for i in range(t["n_layers"])]
    mid = t["n_layers"] - 2
    halo = [int(c) for c in np.flatnonzero(t["layer"] == mid)
            if routine_name(int(t["routine"][c])) == "conv2/igemm_tc" and " halo" in g.candidate_desc(int(c))]
    assert halo, "no halo variant offered"
    ins = [to_device(x, sch)] + ([to_device(r, sch)] if res else [])
    ref = run_layer(layer, [stored_values(x, dt)] + ([stored_values(r, dt)] if res else []), dt)
    for c in halo:
        path = list(io)
        path[mid] = c
        g.set_path(path)
        g.set_option(SN_OPT_CUDA_GRAPH, 0)
        y1 = (g.run_multi(ins)[0] if res else g.run(ins[0])).clone()
        y2 = (g.run_multi(ins)[0] if res else g.run(ins[0])).clone()
        g.set_option(SN_OPT_CUDA_GRAPH, 1)
        y3 = (g.run_multi(ins)[0] if res else g.run(ins[0])).clone()
        torch.cuda.synchronize()
        err = maxrel(from_device(y1, sch), ref)
        assert err <= TOL[dt], (g.candidate_desc(c), err)
        assert torch.equal(y1, y2) and torch.equal(y1, y3), g.candidate_desc(c)
