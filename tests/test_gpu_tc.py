"""Parity of the tcgen05 tensor-core implicit-GEMM routine (NHWC fp16/bf16)
against the oracle, over every routine-parameter combination it offers:
1x1 GEMM tiles, 3x3 stride-1 box tiles, stride-2 sub-lattice maps, channel
counts that are not multiples of the 64-channel K block, output channels
that end inside an epilogue chunk, ragged pixel tiles, CTA-pair tiles whose
second CTA has no pixels, stages of one and of two 64-channel blocks."""
import zlib

import numpy as np
import pytest

import synth
from oracle.net import run_layer
from paper_2110_06037_gb300 import build_graph, routine_name

from gpu_helpers import TOL, from_device, maxrel, stored_values, to_device

pytestmark = pytest.mark.gpu

CASES = [
    # N, C, H, W, K, k, s, pad
    (2, 64, 8, 8, 64, 1, 1, 0),       # plain GEMM, one tile
    (1, 64, 14, 14, 128, 1, 1, 0),    # plain, ragged M (196 rows)
    (2, 128, 7, 7, 256, 1, 1, 0),     # plain, BN 128/256
    (2, 64, 9, 11, 64, 3, 1, 1),      # 3x3 s1, ragged boxes
    (4, 64, 14, 14, 64, 3, 1, 1),
    (2, 128, 8, 8, 192, 3, 1, 1),     # 2 channel blocks, K not a multiple of BN 128
    (2, 64, 16, 16, 128, 3, 2, 1),    # 3x3 s2 (sub-lattice maps)
    (2, 64, 14, 14, 256, 1, 2, 0),    # 1x1 s2 downsample
    (1, 24, 10, 10, 40, 3, 1, 1),     # C and K not multiples of 64 / 32
    (1, 16, 6, 6, 8, 1, 1, 0),        # tiny
    (1, 96, 12, 12, 72, 5, 1, 2),     # 5x5
    (2, 256, 7, 7, 256, 3, 1, 1),     # few tiles: K-split variants (2, 4) offered
    (4, 512, 7, 7, 136, 1, 1, 0),     # plain GEMM K split, K not a multiple of 32
    (2, 128, 16, 16, 128, 3, 2, 1),   # 3x3 s2 with two 64-channel blocks per pipeline stage
    (2, 256, 14, 14, 512, 1, 2, 0),   # 1x1 s2 downsample, two blocks per stage
]


@pytest.mark.parametrize("case", CASES)
@pytest.mark.parametrize("dt", ["f16", "bf16"])
def test_tc_routine_all_variants(case, dt):
    import torch
    N, C, H, W, K, k, s, pd = case
    schema = (dt, "nhwc")
    rng = np.random.default_rng(zlib.crc32(repr((case, dt)).encode()))
    x = rng.standard_normal((N, C, H, W)).astype(np.float32)
    layer = synth.conv(C, K, k, s, pd, act="relu")
    layer["weight"] = (rng.standard_normal((K, C, k, k)) * np.sqrt(2.0 / (C * k * k))).astype(np.float32)
    layer["bias"] = (rng.standard_normal(K) * 0.1).astype(np.float32)
    ref = run_layer(layer, [stored_values(x, dt)], dt)
    spec = dict(layer, inputs=[-1])
    g = build_graph([spec], x.shape, schema, schema, [schema])
    t = g.cost_table()
    tc = [c for c in range(len(t["cost"])) if routine_name(int(t["routine"][c])) == "conv2/igemm_tc"]
    assert tc, "tensor-core routine not offered"
    xd = to_device(x, schema)
    io_in = int(np.flatnonzero(t["layer"] == 0)[0])
    io_out = int(np.flatnonzero(t["layer"] == 2)[0])
    for c in tc:
        g.set_path([io_in, c, io_out])
        y = g.run(xd)
        torch.cuda.synchronize()
        err = maxrel(from_device(y, schema), ref)
        assert err <= TOL[dt], (int(t["variant"][c]), err)
