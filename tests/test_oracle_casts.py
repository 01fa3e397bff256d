"""Pins for the oracle's IEEE-754 casts and layout permutations.  CPU only.

binary16 is pinned to numpy's float16 conversion (a library routine), and
bfloat16 to torch's CPU conversion; both round to nearest even.  Round trips
are checked exhaustively over all 2^16 patterns.
"""
import numpy as np
import torch

import oracle


def _all16():
    return np.arange(65536, dtype=np.uint32).astype(np.uint16)


def test_f16_exhaustive_roundtrip_and_widening():
    h = _all16()
    f = oracle.f16_bits_to_f32(h)
    ref = h.view(np.float16).astype(np.float32)
    nan = np.isnan(ref)
    np.testing.assert_array_equal(np.isnan(f), nan)
    np.testing.assert_array_equal(f[~nan], ref[~nan])
    back = oracle.f32_to_f16_bits(f)
    np.testing.assert_array_equal(back[~nan], h[~nan])
    assert np.all(np.isnan(oracle.f16_bits_to_f32(back[nan])))


def test_bf16_exhaustive_roundtrip_and_widening():
    h = _all16()
    f = oracle.bf16_bits_to_f32(h)
    ref = (h.astype(np.uint32) << 16).view(np.float32)  # bf16 is the top half of fp32
    nan = np.isnan(ref)
    np.testing.assert_array_equal(f[~nan], ref[~nan])
    back = oracle.f32_to_bf16_bits(f)
    np.testing.assert_array_equal(back[~nan], h[~nan])


def _f16_midpoints():
    v = np.arange(0, 0x7c00, dtype=np.uint32).astype(np.uint16).view(np.float16)
    v = v.astype(np.float64)
    mids = (v[:-1] + v[1:]) / 2  # exact in fp32 (12 significant bits)
    return np.concatenate([mids, -mids]).astype(np.float32)


def test_f16_rne_matches_numpy():
    rng = np.random.default_rng(0)
    x = np.concatenate([
        rng.standard_normal(200000).astype(np.float32) * np.float32(3.0),
        (rng.standard_normal(100000) * 1e-6).astype(np.float32),  # subnormal range
        (rng.standard_normal(100000) * 6e4).astype(np.float32),   # overflow edge
        _f16_midpoints(),
        np.array([65504, 65519.996, 65520, 65536, 1e9, -65520, 2 ** -24, 2 ** -25,
                  3 * 2 ** -25, 2 ** -26, 0.0, -0.0, np.inf, -np.inf], np.float32),
    ])
    got = oracle.f32_to_f16_bits(x)
    with np.errstate(over="ignore"):
        ref = x.astype(np.float16).view(np.uint16)
    np.testing.assert_array_equal(got, ref)


def test_f16_hand_cases():
    c = oracle.f32_to_f16_bits(np.array([65504, 65520, 2 ** -24, 2 ** -25, 3 * 2 ** -25,
                                         1 + 2 ** -11, 1 + 3 * 2 ** -11], np.float32))
    # max finite; first value that rounds to inf; min subnormal; tie -> even (0);
    # tie between 1 and 2 quanta -> 2; tie above 1.0 -> 1.0; tie -> 1 + 2^-9
    assert list(c) == [0x7bff, 0x7c00, 0x0001, 0x0000, 0x0002, 0x3c00, 0x3c02]


def test_bf16_rne_matches_torch():
    rng = np.random.default_rng(1)
    base = rng.standard_normal(200000).astype(np.float32)
    mids = ((_all16()[:0x7f80].astype(np.uint32) << 16) | 0x8000).view(np.float32)  # exact ties
    x = np.concatenate([base, base * np.float32(1e30), base * np.float32(1e-38), mids, -mids,
                        np.array([3.3895314e38, 3.3961e38, 0.0, -0.0, np.inf], np.float32)])
    got = oracle.f32_to_bf16_bits(x)
    ref = torch.from_numpy(x).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    np.testing.assert_array_equal(got, ref)


def test_nan_stays_nan():
    x = np.array([np.nan, -np.nan], np.float32)
    assert np.all(np.isnan(oracle.f16_bits_to_f32(oracle.f32_to_f16_bits(x))))
    assert np.all(np.isnan(oracle.bf16_bits_to_f32(oracle.f32_to_bf16_bits(x))))


def test_layout_roundtrip_and_transpose():
    rng = np.random.default_rng(2)
    for dt in (np.float32, np.uint16):
        x = (rng.standard_normal((2, 5, 3, 7)) * 1000).astype(dt)
        y = oracle.nchw_to_nhwc(x)
        np.testing.assert_array_equal(y, x.transpose(0, 2, 3, 1))
        np.testing.assert_array_equal(oracle.nhwc_to_nchw(y), x)
