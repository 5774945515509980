"""Pins of the oracle's 4-bit weights (Section 3: dequantize, add noise, quantize)."""
import numpy as np
import pytest
from scipy import stats

import oracle
import synthetic


def test_levels_are_normal_quantiles():
    """16 levels: quantiles of N(0,1) at the stated probabilities, scaled to [-1, 1]."""
    d = 1 / 32
    neg = stats.norm.ppf(d + (0.5 - d) * np.arange(8) / 7)
    pos = stats.norm.ppf(0.5 + (0.5 - d) * np.arange(1, 9) / 8)
    v = np.concatenate([neg, pos])
    v[7] = 0.0
    want = (v / v[-1]).astype(np.float32)
    got = oracle.q4_levels()
    assert np.array_equal(got, want)
    assert got[0] == -1 and got[7] == 0 and got[15] == 1 and np.all(np.diff(got) > 0)


def _nearest(x, lev):
    d = np.abs(x[:, None] - lev[None, :].astype(np.float64))
    return np.argmin(d, axis=1)  # first minimum: ties go to the lower level


def test_quantize_is_nearest_level_and_absmax():
    w = synthetic.normal_values(64 * 50 + 17, 0.02, 60).astype(np.float64)
    w[:64] = 0.0                       # an all-zero block
    codes, scale = oracle.q4_quantize(w)
    lev = oracle.q4_levels()
    n = w.size
    c = np.empty(n, dtype=np.int64)
    c[0::2] = codes[: (n + 1) // 2] & 0xF
    c[1::2] = codes[: n // 2] >> 4
    for b in range(scale.size):
        blk = w[64 * b: 64 * b + 64]
        assert scale[b] == np.float32(np.abs(blk).max())
        x = blk / scale[b] if scale[b] > 0 else np.zeros_like(blk)
        assert np.array_equal(c[64 * b: 64 * b + blk.size], _nearest(x, lev))
    assert np.all(c[:64] == 7)


def test_quantize_round_trip_and_nibbles():
    w = synthetic.normal_values(64 * 9, 1.0, 61).astype(np.float64)
    codes, scale = oracle.q4_quantize(w)
    back = oracle.q4_dequantize(codes, scale, w.size)
    c2, s2 = oracle.q4_quantize(back)
    assert np.array_equal(codes, c2) and np.array_equal(scale, s2)
    # element 2i in the low nibble of byte i
    lev = oracle.q4_levels()
    one = np.zeros(4)
    one[1] = 1.0  # element 1 -> level 15 in the high nibble of byte 0, the rest -> zero level 7
    c, s = oracle.q4_quantize(one)
    assert c[0] == (15 << 4) | 7 and c[1] == (7 << 4) | 7 and s[0] == 1.0


def test_perturb_zero_eps_identity_and_values():
    w = synthetic.normal_values(64 * 20 + 5, 0.02, 62).astype(np.float64)
    codes, scale = oracle.q4_quantize(w)
    c, s, v = oracle.q4_perturb(codes, scale, w.size, 1024, (3, 1, 0), 0.0)
    assert np.array_equal(c, codes) and np.array_equal(s, scale)
    c, s, v = oracle.q4_perturb(codes, scale, w.size, 1024, (3, 1, 0), 1e-3)
    z = oracle.gaussian_range((3, 1, 0), 1024, w.size)
    np.testing.assert_allclose(v, oracle.q4_dequantize(codes, scale, w.size) + 1e-3 * z,
                               rtol=0, atol=1e-15)
    cq, sq = oracle.q4_quantize(v)
    assert np.array_equal(c, cq) and np.array_equal(s, sq)
