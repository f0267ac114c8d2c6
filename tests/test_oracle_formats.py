"""Pins for the oracle's number formats (binary16 and OCP FP8 E4M3).

The oracle writes both encoders as the literal nearest-value search over the
format's value table.  These tests pin that search against independent
routines: numpy's float16 cast and torch's float8_e4m3fn cast (both IEEE
round-to-nearest-even), over sweeps that hit every rounding decision: values
just below, at and just above every midpoint between neighbours, in every
binade, both signs, plus the subnormal ranges exhaustively.
"""
import numpy as np
import pytest
import torch

import oracle


def test_f16_decode_all_patterns_match_numpy():
    bits = np.arange(1 << 16, dtype=np.uint32).astype(np.uint16)
    ours = oracle.f16_decode(bits)
    ref = bits.view(np.float16).astype(np.float64)
    nan = np.isnan(ref)
    assert np.array_equal(np.isnan(ours), nan)
    assert np.array_equal(ours[~nan], ref[~nan])
    # signed zero is kept
    assert np.signbit(ours[0x8000]) and not np.signbit(ours[0])


def test_f16_encode_roundtrip_every_finite_pattern():
    bits = np.arange(1 << 16, dtype=np.uint32).astype(np.uint16)
    vals = bits.view(np.float16)
    fin = np.isfinite(vals)
    enc = oracle.f16_encode(vals[fin].astype(np.float64))
    assert np.array_equal(enc, bits[fin])


def _midpoint_sweep_f32(low_bits: int) -> np.ndarray:
    """fp32 values whose bits below the target precision sit at, just below
    and just above the rounding midpoint (and at 0 / all-ones), for every
    combination of the higher bits."""
    hi = np.arange(1 << (32 - low_bits), dtype=np.uint64) << np.uint64(low_bits)
    half = 1 << (low_bits - 1)
    lows = np.array([0, 1, half - 1, half, half + 1, (1 << low_bits) - 1], np.uint64)
    pats = (hi[:, None] | lows[None, :]).ravel().astype(np.uint32)
    v = pats.view(np.float32)
    return v[np.isfinite(v)]


def _midpoint_sweeps(first: int, last: int) -> np.ndarray:
    """Midpoint sweeps for every rounding position first..last (subnormal
    targets round at higher bit positions than normal ones)."""
    return np.concatenate([_midpoint_sweep_f32(b) for b in range(first, last + 1)])


def test_f16_encode_matches_numpy_cast_on_midpoints():
    # fp32 has 13 more fraction bits than fp16: sweep every midpoint pattern.
    v = _midpoint_sweep_f32(13)
    ours = oracle.f16_encode(v.astype(np.float64))
    with np.errstate(over="ignore"):
        ref = v.astype(np.float16).view(np.uint16)
    assert np.array_equal(ours, ref)


def test_f16_encode_matches_numpy_cast_on_subnormal_midpoints():
    # fp16 subnormals round at fp32 bit positions 14..23.
    v = _midpoint_sweeps(14, 23)
    v = v[np.abs(v) < 2.0 ** -13]
    ours = oracle.f16_encode(v.astype(np.float64))
    assert np.array_equal(ours, v.astype(np.float16).view(np.uint16))


def test_f16_encode_matches_numpy_cast_exhaustive_slice():
    # Every fp32 bit pattern in [2^-25, 2^-23] and in [1, 1 + 2^-9).
    for a, b in ((2.0 ** -25, 2.0 ** -23), (1.0, 1.0 + 2.0 ** -9)):
        pats = np.arange(np.float32(a).view(np.uint32), np.float32(b).view(np.uint32) + 1,
                         dtype=np.uint32)
        v = pats.view(np.float32)
        assert np.array_equal(oracle.f16_encode(v.astype(np.float64)),
                              v.astype(np.float16).view(np.uint16))


def test_f16_encode_overflow_and_nan():
    assert oracle.f16_encode([65504.0, 65519.99, 65520.0, 1e9, -65520.0]).tolist() == \
        [0x7BFF, 0x7BFF, 0x7C00, 0x7C00, 0xFC00]
    assert oracle.f16_encode([float("nan")])[0] & 0x7C00 == 0x7C00


def test_e4m3_decode_all_codes_match_torch():
    codes = np.arange(256, dtype=np.uint8)
    ours = oracle.e4m3_decode(codes)
    ref = torch.from_numpy(codes).view(torch.float8_e4m3fn).float().double().numpy()
    nan = np.isnan(ref)
    assert nan.sum() == 2  # 0x7F and 0xFF only
    assert np.array_equal(np.isnan(ours), nan)
    assert np.array_equal(ours[~nan], ref[~nan])
    assert ours[0x7E] == 448.0 and ours[0x01] == 2.0 ** -9 and ours[0x08] == 2.0 ** -6


def _torch_e4m3(v: np.ndarray) -> np.ndarray:
    return torch.from_numpy(v).to(torch.float8_e4m3fn).view(torch.uint8).numpy()


def test_e4m3_encode_matches_torch_on_midpoints_in_range():
    # E4M3 keeps 3 fraction bits: sweep the 20 bits below them at/around the
    # midpoint for every sign/exponent/top-mantissa combination.  torch turns
    # magnitudes >= 464 into NaN (no saturation), so compare below 464 only.
    v = _midpoint_sweep_f32(20)
    v = v[np.abs(v) < 464.0]
    assert np.array_equal(oracle.e4m3_encode(v), _torch_e4m3(v))


def test_e4m3_encode_matches_torch_subnormal_midpoints():
    # E4M3 subnormals round at fp32 bit positions 21..23 (and above for the
    # values that round to zero or to the smallest subnormal).
    v = _midpoint_sweeps(21, 26)
    v = v[np.abs(v) < 2.0 ** -5]
    assert np.array_equal(oracle.e4m3_encode(v), _torch_e4m3(v))


def test_e4m3_encode_matches_torch_exhaustive_slice():
    # Every fp32 bit pattern in [2^-11, 2^-9] (round-to-zero edge and the
    # first subnormal) and in [1, 1.25]; both signs.
    for a, b in ((2.0 ** -11, 2.0 ** -9), (1.0, 1.25)):
        pats = np.arange(np.float32(a).view(np.uint32), np.float32(b).view(np.uint32) + 1,
                         dtype=np.uint32)
        v = pats.view(np.float32)
        assert np.array_equal(oracle.e4m3_encode(v), _torch_e4m3(v))
        assert np.array_equal(oracle.e4m3_encode(-v), _torch_e4m3(-v))


def test_e4m3_encode_random_patterns_match_torch():
    rng = np.random.default_rng(7)
    pats = rng.integers(0, 1 << 32, size=1 << 20, dtype=np.uint64).astype(np.uint32)
    v = pats.view(np.float32)
    v = v[np.isfinite(v) & (np.abs(v) < 464.0)]
    assert np.array_equal(oracle.e4m3_encode(v), _torch_e4m3(v))


def test_e4m3_encode_saturates_and_keeps_sign():
    got = oracle.e4m3_encode(np.array([448.0, 463.9, 464.0, 1e30, -1e30, 0.0, -0.0], np.float32))
    assert got.tolist() == [0x7E, 0x7E, 0x7E, 0x7E, 0xFE, 0x00, 0x80]


@pytest.mark.parametrize("x,code", [
    (1.0, 0x38), (-2.0, 0xC0), (17.0, 0x58), (19.0, 0x5A),   # ties go to the even mantissa
    (2.0 ** -9, 0x01), (3 * 2.0 ** -10, 0x02), (2.0 ** -10, 0x00),
    (0.875 * 2.0 ** -6, 0x07), (240.0, 0x77), (0.1, 0x1D),
])
def test_e4m3_encode_hand_values(x, code):
    # value = (8 + m) * 2^(e - 10) for exponent field e >= 1.
    # 17 lies halfway between 16 (0x58) and 18 (0x59): even -> 16.
    # 19 lies halfway between 18 (0x59) and 20 (0x5A): even -> 20.
    # 3*2^-10 lies halfway between 2^-9 (0x01) and 2^-8 (0x02): even -> 0x02.
    # 2^-10 lies halfway between 0 and 2^-9: even -> 0.
    # 0.1 = 1.6 * 2^-4: neighbours 1.625*2^-4 (0x1D) and 1.5*2^-4; nearer 0x1D.
    assert int(oracle.e4m3_encode(np.array([x], np.float32))[0]) == code
