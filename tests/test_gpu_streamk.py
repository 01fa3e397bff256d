"""Stream-K routine parameters of conv2/igemm_tc.

A stream-K variant cuts the layer's tiles' K steps, laid end to end, into one
equal range per SM; a tile whose K steps fall in several ranges is summed from
fp32 parts by the epilogue warp that arrives last at the tile's counter.  On
layers with few tiles (so that every tile is split, some into nine parts of
one K step), ragged pixel counts, an output-channel count that is not a
multiple of the tile, stride 2 and a fused residual input:
  * every stream-K variant matches the oracle within the fp16/bf16 tolerance;
  * a second launch and a CUDA-graph replay give the same bits (the counters
    are left zeroed, and the parts are summed in a fixed order);
  * after a launch stopped by an expired wait, the graph's counters are
    cleared and the next run gives the same bits again.
"""
import numpy as np
import pytest

import synth
from oracle.net import run_layer
from paper_2110_06037_gb300 import (SN_OPT_CHECK, SN_OPT_CUDA_GRAPH, SN_OPT_WAIT_LIMIT, SnError, _sn, build_graph,
                                    routine_name)

from gpu_helpers import TOL, from_device, maxrel, stored_values, to_device

pytestmark = pytest.mark.gpu

# (N, H, C, K, k, stride, residual, dtype)
CASES = [
    (2, 14, 64, 128, 3, 1, False, "bf16"),    # 4 tiles of 9 K steps: one step per CTA
    (4, 28, 128, 256, 3, 2, True, "f16"),     # stride 2, fused residual
    (3, 13, 256, 320, 1, 1, True, "bf16"),    # 507 pixels, 320 channels: ragged in both
    (8, 7, 512, 512, 3, 1, False, "bf16"),    # a ResNet-50 stage-4 layer at batch 8
    (32, 14, 1024, 256, 1, 1, False, "f16"),  # a ResNet-50 stage-3 reduction at batch 32
]


def _graph(N, H, C, K, k, s, res, dt, seed):
    rng = np.random.default_rng(seed)
    layer = synth.conv(C, K, k, s, k // 2, act="relu")
    layer["weight"] = (rng.standard_normal((K, C, k, k)) * np.sqrt(2.0 / (C * k * k))).astype(np.float32)
    layer["bias"] = (rng.standard_normal(K) * 0.1).astype(np.float32)
    P = (H + 2 * (k // 2) - k) // s + 1
    x = rng.standard_normal((N, C, H, H)).astype(np.float32)
    r = rng.standard_normal((N, K, P, P)).astype(np.float32) if res else None
    sch = (dt, "nhwc")
    g = build_graph([dict(layer, inputs=[-1, -2] if res else [-1])], x.shape, sch, sch, [sch],
                    extra_inputs=[(N, K, P, P)] if res else ())
    return g, layer, x, r, sch


def _streamk(g):
    t = g.cost_table()
    io = [int(np.flatnonzero(t["layer"] == i)[0]) for i in range(t["n_layers"])]
    mid = t["n_layers"] - 2
    sk = [int(c) for c in np.flatnonzero(t["layer"] == mid)
          if routine_name(int(t["routine"][c])) == "conv2/igemm_tc" and "streamk" in g.candidate_desc(int(c))]
    return io, mid, sk


def _run(g, ins, res):
    return g.run_multi(ins)[0] if res else g.run(ins[0])


@pytest.mark.parametrize("case", CASES, ids=lambda c: "n%d_h%d_%d-%d_k%ds%d%s_%s" % (
    c[0], c[1], c[2], c[3], c[4], c[5], "_res" if c[6] else "", c[7]))
def test_streamk_variants_match_oracle_and_repeat_bit_for_bit(case):
    import torch
    N, H, C, K, k, s, res, dt = case
    g, layer, x, r, sch = _graph(*case, seed=N * 100 + C + K)
    io, mid, sk = _streamk(g)
    assert sk, "no stream-K variant offered"
    ins = [to_device(x, sch)] + ([to_device(r, sch)] if res else [])
    ref = run_layer(layer, [stored_values(x, dt)] + ([stored_values(r, dt)] if res else []), dt)
    for c in sk:
        path = list(io)
        path[mid] = c
        g.set_path(path)
        g.set_option(SN_OPT_CUDA_GRAPH, 0)
        y1 = _run(g, ins, res).clone()
        y2 = _run(g, ins, res).clone()
        g.set_option(SN_OPT_CUDA_GRAPH, 1)
        y3 = _run(g, ins, res).clone()
        torch.cuda.synchronize()
        err = maxrel(from_device(y1, sch), ref)
        assert err <= TOL[dt], (g.candidate_desc(c), err)
        assert torch.equal(y1, y2) and torch.equal(y1, y3), g.candidate_desc(c)


def test_streamk_counters_are_cleared_after_an_expired_wait():
    import torch
    g, layer, x, r, sch = _graph(2, 14, 64, 128, 3, 1, False, "bf16", seed=5)
    io, mid, sk = _streamk(g)
    path = list(io)
    path[mid] = sk[0]
    g.set_path(path)
    g.set_option(SN_OPT_CHECK, 1)
    g.set_option(SN_OPT_CUDA_GRAPH, 0)
    xd = to_device(x, sch)
    y0 = g.run(xd).clone()
    g.set_option(SN_OPT_WAIT_LIMIT, 1)
    with pytest.raises(SnError) as e:
        g.run(xd)
    assert e.value.status == _sn.SN_ETIMEOUT
    g.set_option(SN_OPT_WAIT_LIMIT, 0)
    y1 = g.run(xd)
    torch.cuda.synchronize()
    assert torch.equal(y0, y1)
