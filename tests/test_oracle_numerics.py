"""Pins for the oracle's numerics: closed forms, hand-worked cases, a library
routine on random shapes, and invariants.  CPU only."""
import os

import numpy as np
import pytest
import torch

import oracle
from oracle.net import run_layer

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _golden_grid(name):
    rows = [l.split() for l in open(os.path.join(GOLDEN, name)) if l.strip() and l[0] != "#"]
    return np.array(rows, dtype=np.float64)


def test_all_ones_border_counts():
    y = oracle.conv2d(np.ones((1, 1, 5, 5)), np.ones((1, 1, 3, 3)), pad=(1, 1))
    np.testing.assert_array_equal(y[0, 0], _golden_grid("conv_ones_3x3_pad1.txt"))


def test_all_ones_scales_with_channels():
    C = 7
    y = oracle.conv2d(np.ones((2, C, 5, 5)), np.ones((3, C, 3, 3)), pad=(1, 1))
    for n in range(2):
        for k in range(3):
            np.testing.assert_array_equal(y[n, k], C * _golden_grid("conv_ones_3x3_pad1.txt"))


def test_ramp_closed_form():
    h, w = np.meshgrid(np.arange(6), np.arange(6), indexing="ij")
    x = (h + w).astype(np.float64)[None, None]
    y = oracle.conv2d(x, np.ones((1, 1, 3, 3)))
    np.testing.assert_array_equal(y[0, 0], _golden_grid("conv_ramp_3x3_valid.txt"))


def test_identity_kernel_is_copy():
    rng = np.random.default_rng(1)
    C = 5
    x = rng.standard_normal((2, C, 7, 9))
    w = np.zeros((C, C, 3, 3))
    for c in range(C):
        w[c, c, 1, 1] = 1.0
    np.testing.assert_array_equal(oracle.conv2d(x, w, pad=(1, 1)), x)
    w1 = np.eye(C).reshape(C, C, 1, 1)
    np.testing.assert_array_equal(oracle.conv2d(x, w1), x)


def test_no_kernel_flip():
    # single tap at (r, s) = (0, 2): y[p, q] = x[p - 1, q + 1] (cross-correlation);
    # a flipped kernel would give x[p + 1, q - 1].
    rng = np.random.default_rng(2)
    x = rng.standard_normal((1, 1, 6, 6))
    w = np.zeros((1, 1, 3, 3))
    w[0, 0, 0, 2] = 1.0
    y = oracle.conv2d(x, w, pad=(1, 1))[0, 0]
    xp = np.pad(x[0, 0], 1)
    np.testing.assert_array_equal(y, xp[0:6, 2:8])


def test_stride_two_subsamples():
    rng = np.random.default_rng(3)
    x = rng.standard_normal((1, 2, 9, 8))
    w = np.zeros((2, 2, 3, 3))
    w[0, 0, 1, 1] = w[1, 1, 1, 1] = 1.0
    y = oracle.conv2d(x, w, stride=(2, 2), pad=(1, 1))
    assert y.shape == (1, 2, 5, 4)
    np.testing.assert_array_equal(y, x[:, :, ::2, ::2])


def test_dilation_shifts():
    rng = np.random.default_rng(4)
    x = rng.standard_normal((1, 1, 8, 8))
    w = np.zeros((1, 1, 3, 3))
    w[0, 0, 2, 2] = 1.0
    y = oracle.conv2d(x, w, pad=(2, 2), dil=(2, 2))[0, 0]  # input index p - 2 + 2*2
    xp = np.pad(x[0, 0], ((0, 2), (0, 2)))
    np.testing.assert_array_equal(y, xp[2:10, 2:10])


def test_group_channel_mapping():
    x = np.arange(4 * 3 * 3, dtype=np.float64).reshape(1, 4, 3, 3)
    w = np.zeros((2, 2, 1, 1))
    w[:, 0, 0, 0] = 1.0
    w[:, 1, 0, 0] = 2.0
    y = oracle.conv2d(x, w, groups=2)
    np.testing.assert_array_equal(y[0, 0], x[0, 0] + 2 * x[0, 1])
    np.testing.assert_array_equal(y[0, 1], x[0, 2] + 2 * x[0, 3])


def test_bias_and_activations():
    x = np.linspace(-8, 8, 17).reshape(1, 1, 1, 17)
    w = np.ones((1, 1, 1, 1))
    b = np.array([0.5])
    np.testing.assert_array_equal(oracle.conv2d(x, w, b)[0, 0, 0], x[0, 0, 0] + 0.5)
    np.testing.assert_array_equal(oracle.conv2d(x, w, b, act="relu")[0, 0, 0],
                                  np.maximum(x[0, 0, 0] + 0.5, 0))
    np.testing.assert_array_equal(oracle.conv2d(x, w, b, act="relu6")[0, 0, 0],
                                  np.clip(x[0, 0, 0] + 0.5, 0, 6))


def test_hard_swish_and_hard_sigmoid_closed_forms():
    """MobileNetV3's piecewise-linear activations at their knots and in each
    piece: hswish(x) = x relu6(x + 3) / 6, hsigmoid(x) = relu6(x + 3) / 6."""
    x = np.array([-10.0, -4.0, -3.0, -1.5, 0.0, 1.0, 1.5, 3.0, 4.0, 10.0])
    z = np.zeros_like(x)
    hsw = oracle.add(x, z, act="hswish")
    hsg = oracle.add(x, z, act="hsigmoid")
    np.testing.assert_allclose(hsw, [0.0, 0.0, 0.0, -0.375, 0.0, 2.0 / 3.0, 1.125, 3.0, 4.0, 10.0], rtol=0, atol=1e-15)
    np.testing.assert_allclose(hsg, [0.0, 0.0, 0.0, 0.25, 0.5, 2.0 / 3.0, 0.75, 1.0, 1.0, 1.0], rtol=0, atol=1e-15)
    # the two are consistent: hswish = x * hsigmoid
    np.testing.assert_allclose(hsw, x * hsg, rtol=0, atol=1e-15)


def test_mul_scales_each_channel():
    """Per-channel scale: a hand case, then the identity and zero scales."""
    x = np.arange(2 * 3 * 2 * 2, dtype=np.float64).reshape(2, 3, 2, 2)
    s = np.array([[1.0, -2.0, 0.5], [0.0, 3.0, -1.0]])
    y = oracle.mul(x, s)
    assert y[0, 1, 1, 0] == x[0, 1, 1, 0] * -2.0 and y[1, 0, 0, 1] == 0.0 and y[1, 2, 1, 1] == -x[1, 2, 1, 1]
    np.testing.assert_array_equal(oracle.mul(x, np.ones((2, 3, 1, 1))), x)
    np.testing.assert_array_equal(oracle.mul(x, np.zeros((2, 3))), np.zeros_like(x))
    np.testing.assert_array_equal(oracle.mul(x, np.full((2, 3), 2.0), act="relu6"), np.clip(2 * x, 0, 6))


@pytest.mark.parametrize("case", [
    # N, C, H, W, K, R, S, stride, pad, dil, groups
    (1, 3, 11, 13, 4, 3, 3, (1, 1), (1, 1), (1, 1), 1),
    (2, 4, 9, 9, 6, 3, 3, (2, 2), (1, 1), (1, 1), 2),
    (1, 6, 10, 7, 6, 3, 3, (1, 2), (1, 1), (1, 1), 6),
    (2, 3, 17, 17, 5, 7, 7, (2, 2), (3, 3), (1, 1), 1),
    (1, 4, 12, 12, 8, 3, 3, (1, 1), (2, 2), (2, 2), 1),
    (3, 8, 5, 6, 16, 1, 1, (1, 1), (0, 0), (1, 1), 1),
    (1, 8, 7, 7, 4, 1, 1, (2, 2), (0, 0), (1, 1), 1),
    (1, 2, 1, 1, 3, 3, 3, (1, 1), (1, 1), (1, 1), 1),
])
def test_conv_matches_library_fp64(case):
    N, C, H, W, K, R, S, st, pd, dl, g = case
    rng = np.random.default_rng(hash(case) % 2**32)
    x = rng.standard_normal((N, C, H, W))
    w = rng.standard_normal((K, C // g, R, S))
    b = rng.standard_normal(K)
    ref = torch.nn.functional.conv2d(torch.from_numpy(x), torch.from_numpy(w),
                                     torch.from_numpy(b), stride=st, padding=pd,
                                     dilation=dl, groups=g).numpy()
    got = oracle.conv2d(x, w, b, stride=st, pad=pd, dil=dl, groups=g)
    assert got.shape == ref.shape
    np.testing.assert_allclose(got, ref, rtol=1e-12, atol=1e-12)


def test_conv_out_dim_formula():
    assert oracle.conv_out_dim(224, 7, 2, 3) == 112
    assert oracle.conv_out_dim(56, 3, 2, 1) == 28
    assert oracle.conv_out_dim(7, 3, 1, 1) == 7
    assert oracle.conv_out_dim(56, 1, 2, 0) == 28
    assert oracle.conv_out_dim(12, 3, 1, 2, 2) == 12


def test_maxpool_neg_inf_padding_and_library():
    x = -np.arange(1, 17, dtype=np.float64).reshape(1, 1, 4, 4)  # all negative
    y = oracle.maxpool2d(x, (3, 3), (2, 2), (1, 1))
    # zero padding would wrongly give 0 at the borders
    np.testing.assert_array_equal(y[0, 0], [[-1, -2], [-5, -6]])
    rng = np.random.default_rng(5)
    x = rng.standard_normal((2, 3, 113, 113))
    ref = torch.nn.functional.max_pool2d(torch.from_numpy(x), 3, 2, 1).numpy()
    np.testing.assert_array_equal(oracle.maxpool2d(x), ref)


def test_gap_ramp_closed_form():
    H, W = 5, 8
    h, w = np.meshgrid(np.arange(H), np.arange(W), indexing="ij")
    x = np.stack([(h + w), 2 * (h + w)]).astype(np.float64)[None]
    y = oracle.gap(x)
    expect = (H - 1) / 2 + (W - 1) / 2
    np.testing.assert_allclose(y[0, :, 0, 0], [expect, 2 * expect], rtol=0, atol=1e-12)


def test_add_and_relu():
    a = np.array([1.0, -2.0, 3.0])
    b = np.array([-4.0, 1.0, 0.5])
    np.testing.assert_array_equal(oracle.add(a, b), [-3.0, -1.0, 3.5])
    np.testing.assert_array_equal(oracle.add(a, b, "relu"), [0.0, 0.0, 3.5])


def test_dense_matches_matmul_and_childnet():
    rng = np.random.default_rng(6)
    x = rng.standard_normal((3, 64, 1, 1))
    w = rng.standard_normal((10, 64))
    b = rng.standard_normal(10)
    y = oracle.dense(x, w, b)
    np.testing.assert_allclose(y[:, :, 0, 0], x[:, :, 0, 0] @ w.T + b, rtol=1e-12, atol=1e-12)
    # childnet: dense == reshape -> 1x1 conv2 -> reshape (section III-D)
    y2 = oracle.conv2d(x, w.reshape(10, 64, 1, 1), b)
    np.testing.assert_allclose(y, y2, rtol=1e-13, atol=1e-13)


def test_depthwise_is_grouped_conv_with_per_channel_taps():
    rng = np.random.default_rng(7)
    C = 5
    x = rng.standard_normal((1, C, 6, 6))
    w = np.zeros((C, 1, 3, 3))
    for c in range(C):
        w[c, 0, 1, 1] = c + 1.0
    y = oracle.conv2d(x, w, pad=(1, 1), groups=C)
    np.testing.assert_array_equal(y, x * np.arange(1, C + 1).reshape(1, C, 1, 1))


def test_run_layer_rounds_weights_to_schema_dtype():
    w = np.full((1, 1, 1, 1), 1.0 + 2.0 ** -12, np.float32)  # not representable in fp16
    layer = {"type": "conv2", "inputs": [-1], "weight": w, "bias": None,
             "params": dict(c_in=1, c_out=1, kh=1, kw=1, sh=1, sw=1, ph=0, pw=0, groups=1)}
    x = np.ones((1, 1, 1, 1))
    assert run_layer(layer, [x], "f32")[0, 0, 0, 0] == np.float32(1.0 + 2.0 ** -12)
    assert run_layer(layer, [x], "f16")[0, 0, 0, 0] == 1.0
