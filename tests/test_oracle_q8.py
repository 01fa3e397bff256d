"""Pins of the qint8 oracle (section II-C symmetric quantisation) against
brute force on Python integers / fractions, closed forms and the pinned fp64
float oracle.  Scales that are powers of two make every fp32 step exact, so
the expected codes follow from exact rational arithmetic with Python's
round-half-to-even (Fraction.__round__)."""
from __future__ import annotations

from fractions import Fraction

import numpy as np
import pytest

import oracle
from oracle import q8

F32 = np.float32


def _clip(v):
    return max(-127, min(127, v))


def test_quantize_grid_and_dequantize_exact():
    s = 2.0 ** -3
    k = np.arange(-127, 128)
    x = (k * s).astype(F32)
    q = q8.quantize(x, s)
    assert q.dtype == np.int8 and np.array_equal(q.astype(int), k)
    assert np.array_equal(q8.dequantize(q, s), x)


def test_quantize_half_way_goes_to_even():
    s = 0.25
    for k in range(-20, 20):
        x = F32((k + 0.5) * s)
        want = round(Fraction(2 * k + 1, 2))  # half to even
        assert int(q8.quantize(np.array([x]), s)[0]) == want, k


def test_quantize_saturates_symmetric():
    s = 0.5
    x = np.array([1e9, -1e9, 127.4 * s, -127.4 * s, 127.6 * s, -200 * s], F32)
    assert q8.quantize(x, s).astype(int).tolist() == [127, -127, 127, -127, 127, -127]


def test_quantize_roundtrip_error_bound():
    rng = np.random.default_rng(11)
    s = 0.0137
    x = rng.uniform(-127 * s, 127 * s, 5000).astype(F32)
    err = np.abs(q8.dequantize(q8.quantize(x, s), s).astype(np.float64) - x)
    assert err.max() <= 0.5 * s * (1 + 1e-5)
    # a wrong direction of the scale (x * s) or floor instead of round breaks this
    assert np.mean(err) > 0.2 * s


def test_weight_quantisation_per_channel():
    rng = np.random.default_rng(3)
    w = rng.standard_normal((6, 3, 3, 3)).astype(F32)
    w[2] = 0.0
    w[4] *= 100.0
    q, s = q8.quantize_weights(w)
    assert q.shape == w.shape and s.shape == (6,)
    for k in range(6):
        if k == 2:
            assert s[k] == 1.0 and not q[k].any()
            continue
        assert np.abs(q[k].astype(int)).max() == 127
        assert abs(float(s[k]) - np.abs(w[k]).max() / 127) <= 1e-6 * float(s[k])
        err = np.abs(q[k] * np.float64(s[k]) - w[k])
        assert err.max() <= 0.5 * s[k] * (1 + 1e-5)


def _brute_conv(x, w, stride, pad, dil, groups):
    """Python-int cross-correlation, zero padding."""
    n, c, h, wd = x.shape
    k, cg, r, s = w.shape
    p = (h + 2 * pad[0] - dil[0] * (r - 1) - 1) // stride[0] + 1
    q = (wd + 2 * pad[1] - dil[1] * (s - 1) - 1) // stride[1] + 1
    kg = k // groups
    out = np.zeros((n, k, p, q), dtype=object)
    for b in range(n):
        for o in range(k):
            g = o // kg
            for i in range(p):
                for j in range(q):
                    acc = 0
                    for cc in range(cg):
                        for u in range(r):
                            for v in range(s):
                                hh = i * stride[0] - pad[0] + u * dil[0]
                                ww = j * stride[1] - pad[1] + v * dil[1]
                                if 0 <= hh < h and 0 <= ww < wd:
                                    acc += int(x[b, g * cg + cc, hh, ww]) * int(w[o, cc, u, v])
                    out[b, o, i, j] = acc
    return out


def _int_weights(rng, shape):
    """Integer weights whose every output channel reaches |127|, so that the
    per-channel scale is exactly 1 and the codes are the weights."""
    w = rng.integers(-127, 128, shape)
    for k in range(shape[0]):
        w[k].flat[rng.integers(0, w[k].size)] = 127 * (1 if k % 2 else -1)
    return w.astype(F32)


@pytest.mark.parametrize("stride,pad,dil,groups,act,resid", [
    ((1, 1), (1, 1), (1, 1), 1, "none", False),
    ((2, 2), (1, 0), (1, 1), 1, "relu", False),
    ((1, 2), (2, 2), (2, 1), 2, "none", True),
    ((1, 1), (1, 1), (1, 1), 4, "relu", True),  # depthwise
])
def test_conv_matches_integer_brute_force(stride, pad, dil, groups, act, resid):
    rng = np.random.default_rng(5 + groups)
    c, k = 4, 4
    x = rng.integers(-127, 128, (2, c, 5, 6)).astype(np.int8)
    w = _int_weights(rng, (k, c // groups, 3, 3))
    qw, sw = q8.quantize_weights(w)
    assert np.all(sw == 1.0) and np.array_equal(qw.astype(F32), w)
    bias = rng.integers(-500, 500, k).astype(F32)
    s_out = 256.0
    acc = _brute_conv(x, qw, stride, pad, dil, groups)
    qr = rng.integers(-127, 128, acc.shape).astype(np.int8) if resid else None
    got = q8.conv2d(x, 1.0, qw, sw, bias, s_out, stride, pad, dil, groups, act,
                    resid=(qr, 1.0) if resid else None)
    want = np.zeros(acc.shape, int)
    for idx in np.ndindex(acc.shape):
        y = acc[idx] + int(bias[idx[1]]) + (int(qr[idx]) if resid else 0)
        if act == "relu":
            y = max(y, 0)
        want[idx] = _clip(round(Fraction(y, 256)))
    assert np.array_equal(got.astype(int), want)


def test_conv_tracks_the_fp64_conv_within_half_a_code():
    """General scales: the codes' values are the fp64 convolution of the
    dequantised operands to within s_out/2 plus fp32 rounding."""
    rng = np.random.default_rng(9)
    x = rng.standard_normal((2, 8, 7, 7)).astype(F32)
    w = (0.2 * rng.standard_normal((6, 8, 3, 3))).astype(F32)
    b = rng.standard_normal(6).astype(F32)
    s_x = q8.absmax_scale(x)
    qx = q8.quantize(x, s_x)
    qw, sw = q8.quantize_weights(w)
    ref = oracle.conv2d(q8.dequantize(qx, s_x).astype(np.float64),
                        (qw.astype(np.float64) * sw.astype(np.float64)[:, None, None, None]),
                        b, stride=(1, 1), pad=(1, 1))
    s_out = F32(np.abs(ref).max() / 120)
    got = q8.dequantize(q8.conv2d(qx, s_x, qw, sw, b, s_out, pad=(1, 1)), s_out).astype(np.float64)
    assert np.abs(got - ref).max() <= 0.5 * s_out + 1e-5 * (np.abs(ref).max() + 1)
    # and the codes use the range: not a constant or a sign-flipped copy
    assert np.corrcoef(got.ravel(), ref.ravel())[0, 1] > 0.999


def test_dense_is_the_1x1_conv_and_brute_force():
    rng = np.random.default_rng(2)
    x = rng.integers(-127, 128, (3, 10)).astype(np.int8)
    w = _int_weights(rng, (5, 10))
    qw, sw = q8.quantize_weights(w)
    b = rng.integers(-100, 100, 5).astype(F32)
    got = q8.dense(x, 1.0, qw, sw, b, 64.0, act="relu")
    for n in range(3):
        for o in range(5):
            acc = sum(int(x[n, i]) * int(w[o, i]) for i in range(10)) + int(b[o])
            assert int(got[n, o]) == _clip(round(Fraction(max(acc, 0), 64)))
    conv = q8.conv2d(x.reshape(3, 10, 1, 1), 1.0, qw.reshape(5, 10, 1, 1), sw, b, 64.0, act="relu")
    assert np.array_equal(conv.reshape(3, 5), got)


def test_maxpool_commutes_with_quantisation():
    rng = np.random.default_rng(4)
    qx = rng.integers(-127, 128, (2, 3, 9, 8)).astype(np.int8)
    s = F32(0.03)
    got = q8.maxpool2d(qx, s, s, k=(3, 3), stride=(2, 2), pad=(1, 1))
    ref = oracle.maxpool2d(q8.dequantize(qx, s).astype(np.float64), k=(3, 3), stride=(2, 2), pad=(1, 1))
    assert np.array_equal(q8.dequantize(got, s).astype(np.float64), ref)
    # requantising to a coarser scale halves the codes (power-of-two ratio)
    half = q8.maxpool2d(qx, 1.0, 2.0, k=(3, 3), stride=(2, 2), pad=(1, 1))
    m = np.rint(q8.dequantize(got, s) / s).astype(int)
    assert np.array_equal(half.astype(int), np.vectorize(lambda v: round(Fraction(int(v), 2)))(m))


def test_gap_exact_mean():
    rng = np.random.default_rng(6)
    qx = rng.integers(-127, 128, (2, 5, 4, 4)).astype(np.int8)
    got = q8.gap(qx, 0.25, 0.25)
    assert got.shape == (2, 5, 1, 1)
    for n in range(2):
        for c in range(5):
            tot = int(qx[n, c].astype(int).sum())
            assert int(got[n, c, 0, 0]) == _clip(round(Fraction(tot, 16)))


def test_add_and_mul_exact():
    rng = np.random.default_rng(8)
    a = rng.integers(-127, 128, (2, 3, 4, 4)).astype(np.int8)
    b = rng.integers(-127, 128, (2, 3, 4, 4)).astype(np.int8)
    got = q8.add(a, 0.5, b, 0.25, 1.0, act="relu")
    want = np.vectorize(lambda u, v: _clip(round(Fraction(max(2 * int(u) + int(v), 0), 4))))(a, b)
    assert np.array_equal(got.astype(int), want)
    sc = rng.integers(-127, 128, (2, 3)).astype(np.int8)
    got = q8.mul(a, 0.5, sc, 2.0 ** -6, 2.0 ** -4)
    for idx in np.ndindex(a.shape):
        y = Fraction(int(a[idx]), 2) * Fraction(int(sc[idx[0], idx[1]]), 64)
        assert int(got[idx]) == _clip(round(y * 16))


def test_hard_activations_closed_forms():
    y = np.array([-4, -3, 0, 1.5, 3, 5], F32)
    assert q8.act_f32(y, "hswish").tolist() == [0, 0, 0, 1.5 * 4.5 / 6, 3, 5]
    assert q8.act_f32(y, "hsigmoid").tolist() == [0, 0, 0.5, F32(4.5) / F32(6), 1, 1]
    assert q8.act_f32(y, "relu6").tolist() == [0, 0, 0, 1.5, 3, 5]


def test_qint8_net_tracks_the_float_net():
    """A small conv-pool-dense net run end to end on codes stays within a few
    output codes of the fp64 float net (the quantisation error budget)."""
    from oracle.net import run_net
    rng = np.random.default_rng(12)
    layers = [
        {"type": "conv2", "inputs": [-1], "params": dict(c_in=3, c_out=8, kh=3, kw=3, sh=1, sw=1, ph=1, pw=1,
                                                         act="relu"),
         "weight": (0.3 * rng.standard_normal((8, 3, 3, 3))).astype(F32),
         "bias": (0.1 * rng.standard_normal(8)).astype(F32)},
        {"type": "maxpool", "inputs": [0], "params": dict(kh=2, kw=2, sh=2, sw=2, ph=0, pw=0)},
        {"type": "gap", "inputs": [1]},
        {"type": "dense", "inputs": [2], "params": dict(act="none"),
         "weight": (0.3 * rng.standard_normal((4, 8))).astype(F32), "bias": np.zeros(4, F32)},
    ]
    x = rng.standard_normal((2, 3, 8, 8)).astype(F32)
    s_in, scales = q8.calibrate(layers, x)
    ref = run_net(layers, x)
    got = q8.run_net_q8(layers, x, s_in, scales)
    assert got.shape == ref.reshape(2, 4).shape or got.shape == ref.shape
    err = np.abs(got.reshape(ref.shape).astype(np.float64) - ref)
    assert err.max() <= 4 * float(scales[-1]) + 1e-6


def test_fused_dequantisation_output_is_the_unrounded_value():
    """A qint8 routine that writes a float schema leaves act(conv + bias) in
    that dtype instead of requantising: with unit scales and integer weights
    that is the exact integer sum (no division by the output scale)."""
    rng = np.random.default_rng(19)
    x = rng.integers(-127, 128, (1, 4, 5, 5)).astype(np.int8)
    w = _int_weights(rng, (3, 4, 3, 3))
    qw, sw = q8.quantize_weights(w)
    b = rng.integers(-50, 50, 3).astype(F32)
    got = q8.conv2d(x, 1.0, qw, sw, b, 256.0, pad=(1, 1), act="relu", out_dtype="f32")
    acc = _brute_conv(x, qw, (1, 1), (1, 1), (1, 1), 1)
    want = np.vectorize(lambda v: float(v))(acc).astype(np.float64) + b.reshape(1, 3, 1, 1)
    assert np.array_equal(got.astype(np.float64), np.maximum(want, 0))
    # and in fp16 it is that value rounded to nearest even
    h = q8.conv2d(x, 1.0, qw, sw, b, 256.0, pad=(1, 1), act="relu", out_dtype="f16")
    assert np.array_equal(h, oracle.round_to(got.astype(np.float32), "f16"))
    # requantising it gives the ordinary qint8 output
    assert np.array_equal(q8.requantize(got, 256.0), q8.conv2d(x, 1.0, qw, sw, b, 256.0, pad=(1, 1), act="relu"))


def test_absmax_scale_hand_cases():
    """Calibration scale = max |x| / 127 in fp32 (section II-C, symmetric),
    1 for an all-zero (or empty) blob.  127 and 254 give exactly 1 and 2."""
    assert q8.absmax_scale(np.array([-127.0, 3.0, 50.0], F32)) == F32(1.0)
    assert q8.absmax_scale(np.array([[1.0, 254.0], [-2.0, 0.5]], F32)) == F32(2.0)
    # the magnitude counts, not the sign: the largest entry is negative
    assert q8.absmax_scale(np.array([12.7, -25.4], F32)) == F32(25.4) / F32(127)
    assert q8.absmax_scale(np.zeros((2, 3), F32)) == F32(1.0)
    assert q8.absmax_scale(np.zeros((0,), F32)) == F32(1.0)
    assert q8.absmax_scale(np.array([-0.0, 0.0], F32)) == F32(1.0)


def test_calibrate_scales_each_blob_by_its_own_maximum():
    """One float pass of a 3-layer net whose blobs have hand-known maxima:
    x has max |x| = 127 * 4; an identity 1x1 conv (+ReLU) keeps the positive
    part (max 127 * 3); a 2x2 max pool keeps that maximum; a GAP of the conv
    output averages channel 0 to (381 + 1 + 2 + 0) / 4 = 96 and channel 1 to
    254.  Scales: input 4, then 3, 3 and 2 in layer order (an off-by-one blob
    index or a missing /127 changes one of them)."""
    x = np.zeros((1, 2, 2, 2), F32)
    x[0, 0] = [[127 * 3, 1], [2, -127 * 4]]      # channel 0: max |.| = 508, max(.) = 381
    x[0, 1] = [[254, 254], [254, 254]]           # channel 1: constant 254
    eye = np.eye(2, dtype=F32).reshape(2, 2, 1, 1)
    layers = [
        {"type": "conv2", "inputs": [-1], "params": dict(c_in=2, c_out=2, kh=1, kw=1, sh=1, sw=1, ph=0, pw=0,
                                                         act="relu"),
         "weight": eye, "bias": np.zeros(2, F32)},
        {"type": "maxpool", "inputs": [0], "params": dict(kh=2, kw=2, sh=2, sw=2, ph=0, pw=0)},
        {"type": "gap", "inputs": [0]},
    ]
    s_in, scales = q8.calibrate(layers, x)
    assert s_in == F32(4.0)
    # conv + ReLU: channel 0 max 381 (= 127 * 3), channel 1 254 -> blob max 381
    assert scales[0] == F32(3.0)
    # pool of a 2x2 map to 1x1: the maxima 381 and 254 -> blob max 381
    assert scales[1] == F32(3.0)
    # GAP of the conv output: channel means 96 and 254 -> blob max 254
    assert scales[2] == F32(2.0)
    # and a blob that is all zero gets scale 1
    x0 = np.zeros_like(x)
    s0, sc0 = q8.calibrate(layers, x0)
    assert s0 == F32(1.0) and all(s == F32(1.0) for s in sc0)
