"""Pins for the oracle's quantizers (Sec. III-A.1 Q4 = f(W16,4), Sec. III-A.2 Q8 = f(W16,8)).

* hand-derived golden fixtures (tests/golden/int4_hand.json, fp8_hand.json);
* INT4: the stored code is the brute-force nearest of the 16 codes to w
  (exact distance |w - c s|, ties to the even code) for every finite fp16 w
  below the group maximum, over a sweep of group maxima; |w - c s| <= s/2;
* FP8: the oracle equals the same scheme composed from torch library
  operations (fp32 divide, torch's E4M3 cast); the error stays within half
  an E4M3 step;
* dequantisation is pinned by an independent decoding of the nibbles.
"""
import json
import os

import numpy as np
import pytest
import torch

import oracle

GOLD = os.path.join(os.path.dirname(__file__), "golden")


def _f16bits(vals):
    return np.asarray(vals, np.float64).astype(np.float16).view(np.uint16)


def _row_from_group(group, fill, width=128):
    row = np.full(width, fill, np.float64)
    row[: len(group)] = group
    return row


def _unpack(codes, K):
    lo = (codes & 0x0F).astype(np.int32) - 8
    hi = (codes >> 4).astype(np.int32) - 8
    out = np.empty((codes.shape[0], K), np.int32)
    out[:, 0::2] = lo
    out[:, 1::2] = hi
    return out


def test_int4_golden_hand_cases():
    d = json.load(open(os.path.join(GOLD, "int4_hand.json")))
    for case in d["cases"]:
        row = _row_from_group(case["group"], case["fill"])
        codes, scales = oracle.quantize_int4(_f16bits(row)[None, :])
        assert int(scales[0, 0]) == case["scale_bits"], case["name"]
        c = _unpack(codes, 128)[0]
        n = len(case["group"])
        assert c[:n].tolist() == case["codes"], case["name"]
        assert (c[n:] == case["fill_code"]).all(), case["name"]


def test_int4_nibble_order_low_nibble_is_even_k():
    row = np.zeros(256)
    row[0], row[1], row[128], row[255] = 7.0, -3.0, 1.0, 7.0
    codes, scales = oracle.quantize_int4(_f16bits(row)[None, :])
    assert codes.shape == (1, 128) and scales.shape == (1, 2)
    assert codes[0, 0] == ((-3 + 8) << 4) | (7 + 8)
    # second group: amax 7 -> s = 1; w[128] = 1 -> code 1 in the low nibble of byte 64
    assert codes[0, 64] & 0x0F == 1 + 8
    assert codes[0, 127] >> 4 == 7 + 8


def _all_finite_f16():
    bits = np.arange(1 << 16, dtype=np.uint32).astype(np.uint16)
    v = bits.view(np.float16)
    return v[np.isfinite(v)].astype(np.float64)


@pytest.mark.parametrize("amax", [
    2.0 ** -24, 3 * 2.0 ** -24, 5 * 2.0 ** -24, 2.0 ** -20, 1e-3, 0.0999755859375,
    0.02, 0.06, 0.5, 1.0, 7.0, 7.5, 100.0, 1000.0, 65504.0,
])
def test_int4_codes_are_bruteforce_nearest(amax):
    amax = float(np.float16(amax))
    allv = _all_finite_f16()
    vals = allv[np.abs(allv) <= amax]
    # every group holds amax first, so every group's scale is the same s
    per = 127
    ngroups = (len(vals) + per - 1) // per
    padded = np.zeros(ngroups * per)
    padded[: len(vals)] = vals
    groups = np.concatenate([np.full((ngroups, 1), amax), padded.reshape(ngroups, per)], axis=1)
    K = 128 * 8
    rows = (ngroups + 7) // 8
    W = np.zeros((rows * 8, 128))
    W[:ngroups] = groups
    W = W.reshape(rows, K)
    codes, scales = oracle.quantize_int4(_f16bits(W))
    s = oracle.f16_decode(scales).reshape(-1)[:ngroups]
    assert np.all(s == s[0])
    s = s[0]
    c = _unpack(codes, K).reshape(-1, 128)[:ngroups, 1:].reshape(-1)[: len(vals)]
    if s == 0:
        assert (c == 0).all()
        return
    # brute force: distances to all 16 codes, exact in double (short dyadics)
    cand = np.arange(-8, 8)
    dist = np.abs(vals[:, None] - cand[None, :] * s)
    best = dist.min(axis=1, keepdims=True)
    tie_ok = dist == best
    # among tied candidates, the even code wins
    even_pick = np.where(tie_ok & (cand[None, :] % 2 == 0), cand[None, :], 99).min(axis=1)
    any_pick = np.where(tie_ok, cand[None, :], 99).min(axis=1)
    expected = np.where((tie_ok & (cand[None, :] % 2 == 0)).any(axis=1), even_pick, any_pick)
    assert np.array_equal(c, expected)
    unclamped = np.abs(vals) <= 7.5 * s
    assert np.all(np.abs(vals - c * s)[unclamped] <= s / 2)


def test_int4_scale_is_fp16_of_amax_over_7():
    rng = np.random.default_rng(1)
    W = (rng.standard_normal((64, 1024)) * 0.02).astype(np.float16)
    codes, scales = oracle.quantize_int4(W.view(np.uint16))
    amax = np.abs(W.astype(np.float32)).reshape(64, 8, 128).max(axis=2)
    ref = (amax / np.float32(7.0)).astype(np.float16).view(np.uint16)
    assert np.array_equal(scales, ref)


def test_int4_dequant_matches_independent_decode():
    rng = np.random.default_rng(2)
    W = (rng.standard_normal((16, 512)) * 0.02).astype(np.float16)
    codes, scales = oracle.quantize_int4(W.view(np.uint16))
    deq = oracle.dequant_int4(codes, scales, 512)
    s = np.repeat(scales.view(np.float16).astype(np.float64), 128, axis=1)
    assert np.array_equal(deq, _unpack(codes, 512) * s)
    # quantisation error within half a step everywhere (no clamping at these scales)
    assert np.all(np.abs(W.astype(np.float64) - deq) <= s / 2)


def test_int4_rejects_bad_shapes_and_nonfinite():
    with pytest.raises(ValueError):
        oracle.quantize_int4(np.zeros((2, 100), np.uint16))
    W = np.zeros((1, 128), np.float16)
    W[0, 3] = np.inf
    with pytest.raises(ValueError):
        oracle.quantize_int4(W.view(np.uint16))


def test_fp8_golden_hand_cases():
    d = json.load(open(os.path.join(GOLD, "fp8_hand.json")))
    for case in d["cases"]:
        row = np.asarray(case["row"], np.float64)
        codes, scales = oracle.quantize_fp8(_f16bits(row)[None, :])
        assert float(scales[0]) == case["scale"], case["name"]
        assert codes[0].tolist() == case["codes"], case["name"]


def _torch_fp8_quant(W16: np.ndarray):
    w = torch.from_numpy(W16.astype(np.float32))
    amax = w.abs().amax(dim=1)
    s = amax / torch.tensor(448.0, dtype=torch.float32)
    safe = torch.where(s == 0, torch.ones_like(s), s)
    c = (w / safe[:, None]).to(torch.float8_e4m3fn).view(torch.uint8)
    c = torch.where((s == 0)[:, None], torch.zeros_like(c), c)
    return c.numpy(), s.numpy()


def test_fp8_matches_torch_composed_scheme():
    rng = np.random.default_rng(3)
    W = (rng.standard_normal((128, 896)) * 0.02).astype(np.float16)
    W[5] = 0
    W[7, :] = np.float16(6e-8)
    W[9, 17] = np.float16(-60000.0)
    codes, scales = oracle.quantize_fp8(W.view(np.uint16))
    tc, ts = _torch_fp8_quant(W)
    assert np.array_equal(scales, ts)
    assert np.array_equal(codes, tc)


def test_fp8_error_within_half_step():
    rng = np.random.default_rng(4)
    W = (rng.standard_normal((32, 640)) * 0.02).astype(np.float16)
    codes, scales = oracle.quantize_fp8(W.view(np.uint16))
    deq = oracle.dequant_fp8(codes, scales)
    w = W.astype(np.float64)
    s = scales.astype(np.float64)[:, None]
    t = np.abs(w / s)
    # E4M3 step at magnitude t: 2^(floor(log2 t) - 3) for t >= 2^-6, else 2^-9
    e = np.floor(np.log2(np.maximum(t, 2.0 ** -6)))
    step = np.where(t >= 2.0 ** -6, 2.0 ** (e - 3), 2.0 ** -9)
    # plus the fp32 rounding of w / s (relative 2^-24)
    assert np.all(np.abs(w - deq) <= (step / 2 + t * 2.0 ** -23) * s)
    dec = oracle.e4m3_decode(codes)
    assert np.array_equal(deq, dec * s)
