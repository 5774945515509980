"""Pins of the CPU oracle against facts that do not come from the oracle itself.

Every check here runs on the CPU. Each pins one part of the oracle so that a
plausible slip in it (a wrong word, sign, index, factor or rounding) fails:

* the Philox4x32-10 stream against PyTorch's independent at::Philox4_32 engine;
* the seed -> (key, counter) map and the element -> (block, word) map, also
  against at::Philox4_32 words;
* the uniforms at their closed-form end points;
* Box-Muller by its polar inverse (radius and angle recovered with hypot and
  atan2) and by the moments and CDF of N(0, 1) over many draws;
* bf16 rounding against torch's float -> bfloat16 conversion;
* the perturbation, the update and the SPSA estimator by special cases,
  restoration bounds, linearity and the closed form of a quadratic loss.
"""
import ctypes
import json
import math
import os

import numpy as np
import pytest
import torch

import oracle
import synthetic

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def aten_blocks(lib, seed, first, n):
    mid, step, sample = seed
    out = np.empty((n, 4), dtype=np.uint32)
    lib.aten_philox_blocks(int(mid), int(step) | (int(sample) << 32), int(first), int(n),
                           out.ctypes.data)
    return out


EDGE_SEEDS = [
    (0, 0, 0),
    (0xFFFFFFFFFFFFFFFF, 0xFFFFFFFF, 0xFFFFFFFF),
    (1_700_000_000_000_000_137, 3, 0),
    (0x00000001FFFFFFFF, 0, 7),
    (0xDEADBEEF00000000, 12345, 0xFFFFFFFF),
]


# --- Philox stream ----------------------------------------------------------

@pytest.mark.parametrize("seed", EDGE_SEEDS)
def test_philox_matches_aten_engine(aten_philox, seed):
    for first in (0, 1, 0xFFFFFFFE, 0xFFFFFFFF, 1 << 32, (1 << 33) + 5, 7_493_635_072):
        ref = aten_blocks(aten_philox, seed, first, 3)
        got = oracle.philox_blocks(seed, first, 3)
        assert np.array_equal(ref, got), (seed, first)


def test_philox_matches_aten_random(aten_philox):
    g = synthetic.rng(1)
    for _ in range(200):
        seed = (int(g.integers(0, 2**64, dtype=np.uint64)), int(g.integers(0, 2**32)),
                int(g.integers(0, 2**32)))
        first = int(g.integers(0, 2**40))
        assert np.array_equal(aten_blocks(aten_philox, seed, first, 2),
                              oracle.philox_blocks(seed, first, 2))


def test_philox_raw_counter_layout(aten_philox):
    # philox(ctr, key) with ctr = (b lo, b hi, step, sample), key = (mid lo, mid hi)
    mid, step, sample, b = 0x0123456789ABCDEF, 77, 5, (3 << 32) + 9
    words = oracle.philox([b & 0xFFFFFFFF, b >> 32, step, sample],
                          [mid & 0xFFFFFFFF, mid >> 32])
    assert np.array_equal(words, aten_blocks(aten_philox, (mid, step, sample), b, 1)[0])


# --- uniforms -----------------------------------------------------------------

def test_uniform_endpoints_closed_form():
    assert oracle.uniform_a(0) == 2.0**-24
    assert oracle.uniform_a(0xFFFFFFFF) == 1.0 - 2.0**-24
    assert oracle.uniform_a(0x1FF) == 2.0**-24          # low 9 bits are dropped
    assert oracle.uniform_a(0x200) == 3 * 2.0**-24
    assert oracle.uniform_b(0) == 2.0**-25
    assert oracle.uniform_b(0xFFFFFFFF) == 1.0 - 2.0**-25
    assert oracle.uniform_b(0x80000000) == 0.5 + 2.0**-25
    # every radius uniform is exactly representable in fp32
    for x in (0, 1 << 9, 12345 << 9, 0xFFFFFFFF, 0x80000000, 0x7FFFFFFF):
        u = oracle.uniform_a(x)
        assert float(np.float32(u)) == u


# --- Box-Muller ---------------------------------------------------------------

def _pairs_from_aten(aten_philox, n_blocks):
    w = aten_blocks(aten_philox, (0xA5A5A5A5DEADBEEF, 9, 2), 1000, n_blocks)
    return w.reshape(-1, 2)


def test_box_muller_polar_inverse(aten_philox):
    """hypot(z0, z1)^2 = -2 ln u_a and atan2(z1, z0) = 2 pi u_b (mod 2 pi)."""
    words = _pairs_from_aten(aten_philox, 50000)
    z = oracle.box_muller_pairs(words)
    ua = ((words[:, 0] >> 9).astype(np.float64) + 0.5) * 2.0**-23
    ub = ((words[:, 1] >> 8).astype(np.float64) + 0.5) * 2.0**-24
    r2 = z[:, 0] ** 2 + z[:, 1] ** 2
    np.testing.assert_allclose(r2, -2.0 * np.log(ua), rtol=1e-12, atol=1e-300)
    ang = np.mod(np.arctan2(z[:, 1], z[:, 0]), 2 * np.pi)
    d = np.abs(ang - 2 * np.pi * ub)
    d = np.minimum(d, 2 * np.pi - d)
    assert d.max() < 1e-9


def test_box_muller_quadrants():
    """Angle words in each quarter turn land in that quadrant (signs of cos, sin)."""
    xa = 0x40000000  # u_a ~ 0.25, radius ~ 1.665
    for quarter, (sc, ss) in enumerate([(1, 1), (-1, 1), (-1, -1), (1, -1)]):
        xb = (quarter << 30) | (1 << 29)       # the middle of the quarter turn
        z = oracle.box_muller_pairs(np.array([[xa, xb]], dtype=np.uint32))[0]
        assert np.sign(z[0]) == sc and np.sign(z[1]) == ss
        assert abs(abs(z[0]) - abs(z[1])) < 1e-6  # 45 degrees into the quadrant


def test_gaussian_index_map_against_aten_words(aten_philox):
    """Element e uses block e >> 2; pair (e >> 1) & 1 of it; cos for even e."""
    seed = (0x1234_5678_9ABC_DEF0, 41, 3)
    first_block = (1 << 32) - 2  # crosses the 32-bit block boundary
    words = aten_blocks(aten_philox, seed, first_block, 4)
    zpairs = oracle.box_muller_pairs(words.reshape(-1, 2)).reshape(-1)
    got = oracle.gaussian_range(seed, first_block * 4, 16)
    np.testing.assert_array_equal(got, zpairs)


def _moments_over(n_total, chunk=10_000_000):
    s1 = s2 = s3 = s4 = 0.0
    n = 0
    seeds = [(synthetic.MASTER_SEED + i, i, 2 * i + 1) for i in range(n_total // chunk)]
    for i, sd in enumerate(seeds):
        z = oracle.gaussian_range(sd, i * 7919, chunk)
        s1 += z.sum(); s2 += (z * z).sum(); s3 += (z ** 3).sum(); s4 += (z ** 4).sum()
        n += z.size
    return n, s1 / n, s2 / n, s3 / n, s4 / n


def test_gaussian_moments_1e8():
    """Mean 0, variance 1, skew 0, kurtosis 3 within 5 standard errors."""
    n, m1, m2, m3, m4 = _moments_over(100_000_000)
    var = m2 - m1 * m1
    assert abs(m1) < 5 / math.sqrt(n)
    assert abs(var - 1) < 5 * math.sqrt(2 / n)
    assert abs(m3) < 5 * math.sqrt(15 / n)        # Var(z^3) = 15
    assert abs(m4 - 3) < 5 * math.sqrt(96 / n)    # Var(z^4) = 105 - 9
    # the extreme radius is sqrt(-2 ln 2^-24)
    assert math.isclose(math.sqrt(-2 * math.log(2.0**-24)), math.sqrt(48 * math.log(2)))


def test_gaussian_cdf_ks():
    from scipy import stats
    z = oracle.gaussian_range((77, 1, 0), 0, 2_000_000)
    for part in (z, z[0::2], z[1::2]):
        res = stats.kstest(part, "norm")
        assert res.pvalue > 1e-4, res


def test_gaussian_independence():
    n = 2_000_000
    z = oracle.gaussian_range((5, 0, 0), 0, n)
    # the two members of a Box-Muller pair are uncorrelated, and so are blocks
    for a, b in ((z[0::2], z[1::2]), (z[0::4], z[2::4]), (z[:-1], z[1:])):
        assert abs(np.corrcoef(a, b)[0, 1]) < 5 / math.sqrt(a.size)
    # streams of different machines, steps and samples are uncorrelated
    for other in ((6, 0, 0), (5, 1, 0), (5, 0, 1)):
        w = oracle.gaussian_range(other, 0, n)
        assert abs(np.corrcoef(z, w)[0, 1]) < 5 / math.sqrt(n)
        assert not np.array_equal(z[:64], w[:64])


# --- bf16 rounding ------------------------------------------------------------

def test_round_bf16_matches_torch():
    g = synthetic.rng(2)
    bits = g.integers(0, 2**32, size=200_000, dtype=np.uint64).astype(np.uint32)
    # add exact ties (low half 0x8000), both parities, subnormals, near-overflow
    ties = (bits & 0xFFFF0000) | 0x8000
    special = np.array([0x00000000, 0x80000000, 0x00000001, 0x00008000, 0x00018000,
                        0x007F8000, 0x00800000, 0x7F7F7FFF, 0x7F7F8000, 0x7F7FFFFF,
                        0xFF7F8000, 0x3F808000, 0x3F818000], dtype=np.uint32)
    allbits = np.concatenate([bits, ties, special])
    f = allbits.view(np.float32)
    f = f[np.isfinite(f)]
    ref = torch.from_numpy(f.copy()).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    got = oracle.round_bf16(f.astype(np.float64))
    assert np.array_equal(got, ref)


def test_round_bf16_specials():
    assert oracle.round_bf16([float("inf")])[0] == 0x7F80
    assert oracle.round_bf16([-float("inf")])[0] == 0xFF80
    assert (oracle.round_bf16([float("nan")])[0] & 0x7FFF) > 0x7F80
    assert oracle.round_bf16([1e39])[0] == 0x7F80       # beyond bf16 max
    assert oracle.round_bf16([-0.0])[0] == 0x8000


# --- perturbation -----------------------------------------------------------

def test_perturb_zero_eps_is_identity():
    th = synthetic.normal_values(1000, 0.02, 1)
    assert np.array_equal(oracle.perturb(th, 5, (1, 2, 3), 0.0), th)
    hb = oracle.round_bf16(th.astype(np.float64))
    assert np.array_equal(oracle.perturb(hb, 5, (1, 2, 3), 0.0), hb)


def test_perturb_from_zero_is_scaled_noise():
    seed, off = (99, 4, 1), 123
    z = oracle.gaussian_range(seed, off, 777)
    got = oracle.perturb(np.zeros(777, np.float32), off, seed, 0.25)  # 0.25 z is exact
    assert np.array_equal(got, (0.25 * z).astype(np.float32))
    gotb = oracle.perturb(np.zeros(777, np.uint16), off, seed, 1.0)
    assert np.array_equal(gotb, oracle.round_bf16(z))


def test_perturb_flat_offset_is_global_index():
    """A tensor at flat offset F sees the same noise as elements F.. of one big tensor."""
    seed = (3, 1, 0)
    big = synthetic.normal_values(5000, 0.02, 2)
    whole = oracle.perturb(big, 0, seed, 1e-3)
    for F, n in ((0, 10), (13, 1001), (4096, 904), (4999, 1)):
        part = oracle.perturb(big[F:F + n], F, seed, 1e-3)
        assert np.array_equal(part, whole[F:F + n])


def test_perturb_restore_bound():
    """+eps, -2 eps, +eps (Algorithm 1) restores theta up to three roundings."""
    seed, eps = (11, 0, 0), 1e-3
    th = synthetic.normal_values(100_000, 0.02, 3)
    th[:1000] = 0.0  # zero biases: a relative-only bound fails there
    z = np.abs(oracle.gaussian_range(seed, 0, th.size))
    t = th
    for e in (eps, -2 * eps, eps):
        t = oracle.perturb(t, 0, seed, e)
    scale = np.abs(th.astype(np.float64)) + 2 * eps * z
    ulp = np.spacing(scale.astype(np.float32)).astype(np.float64)
    assert np.all(np.abs(t.astype(np.float64) - th) <= 1.5 * ulp + 1e-45)
    # with one rounding less (f64 storage) the sequence restores almost exactly
    d = oracle.gaussian_range(seed, 0, th.size)
    back = ((th + eps * d) - 2 * eps * d) + eps * d
    assert np.all(np.abs(back - th) <= 1.5 * np.spacing(np.abs(th) + 2 * eps * np.abs(d)))


# --- codec --------------------------------------------------------------------

@pytest.mark.parametrize("S", [1.0, 8.0, 16.0])
def test_codec_round_trip_all_codes(S):
    for q in range(-127, 128):
        assert oracle.quantize(oracle.dequantize(q, S), S) == q
    assert oracle.dequantize(-128, S) == oracle.dequantize(-127, S)
    assert oracle.dequantize(0, S) == 0.0


@pytest.mark.parametrize("S", [1.0, 16.0])
def test_codec_monotone_odd_clipped(S):
    g = np.concatenate([-np.logspace(-6, 60, 3000)[::-1], [0.0], np.logspace(-6, 60, 3000)])
    q = np.array([oracle.quantize(v, S) for v in g])
    assert np.all(np.diff(q) >= 0)
    assert np.array_equal(q, -np.array([oracle.quantize(-v, S) for v in g]))
    assert q.max() == 127 and q.min() == -127
    assert oracle.quantize(0.0, S) == 0
    assert oracle.quantize(float("nan"), S) == 0
    assert oracle.quantize(float("inf"), S) == 127
    assert oracle.quantize(-float("inf"), S) == -127


@pytest.mark.parametrize("S", [1.0, 16.0])
def test_codec_rounding_boundaries(S):
    """ln(1 + |g|) S is rounded half away from zero: boundaries at expm1((n + 1/2)/S)."""
    for n in range(0, 127):
        b = math.expm1((n + 0.5) / S)
        assert oracle.quantize(b * (1 + 1e-12), S) == n + 1
        assert oracle.quantize(b * (1 - 1e-12), S) == n
        assert oracle.quantize(-b * (1 + 1e-12), S) == -(n + 1)


def test_codec_paper_constants():
    with open(os.path.join(GOLDEN, "paper_constants.json")) as f:
        pc = json.load(f)
    clip = pc["byte_clip"]["value"]
    assert oracle.quantize(1e300, 1.0) == clip and oracle.quantize(-1e300, 1.0) == -clip
    assert pc["bytes_per_projected_gradient"]["value"] == np.dtype(np.int8).itemsize


def test_codec_golden_table():
    """Frozen oracle codec values (tests/golden/codec_table.txt, from make_golden.py)."""
    with open(os.path.join(GOLDEN, "codec_table.txt")) as f:
        rows = [ln.split() for ln in f if ln.strip() and not ln.startswith("#")]
    for kind, S, a, b in rows:
        if kind == "deq":
            assert oracle.dequantize(int(a), float(S)) == float.fromhex(b)
        else:
            assert oracle.quantize(float.fromhex(a), float(S)) == int(b)


# --- update -------------------------------------------------------------------

def _seeds(k, step=0):
    mids = synthetic.machine_ids(k, 7)
    return [(int(m), step, 0) for m in mids]


def test_update_k0_identity_and_k1_is_perturb():
    th = synthetic.normal_values(3001, 0.02, 4)
    assert np.array_equal(oracle.update(th, 8, [], [], 1e-3, 1.0, 16.0), th)
    s = _seeds(1)
    for q in (-128, -5, 0, 1, 77, 127):
        c = oracle.coefficient(q, 1e-3, 1.0, 16.0)
        assert np.array_equal(oracle.update(th, 8, s, [q], 1e-3, 1.0, 16.0),
                              oracle.perturb(th, 8, s[0], c))


def test_update_coefficient_is_descent_direction():
    """The update weight of Algorithm 1 is minus gradient times learning rate over
    the number of gradients: a positive gradient gives a negative step."""
    with open(os.path.join(GOLDEN, "paper_constants.json")) as f:
        pc = json.load(f)
    sign = pc["update_weight"]["sign"]
    for q in (1, 50, 127):
        c = oracle.coefficient(q, 1e-2, 4.0, 16.0)
        assert np.sign(c) == sign
        assert c == np.float32(-1e-2 * oracle.dequantize(q, 16.0) / 4.0)
    assert oracle.coefficient(0, 1.0, 1.0, 1.0) == 0.0


def test_update_order_invariant_and_duplicates_rejected():
    th = synthetic.normal_values(2000, 0.02, 5)
    s = _seeds(9)
    q = synthetic.byte_codes(9, 1)
    ref = oracle.update(th, 0, s, q, 1e-4, 9.0, 16.0)
    perm = synthetic.rng(3).permutation(9)
    got = oracle.update(th, 0, [s[i] for i in perm], q[perm], 1e-4, 9.0, 16.0)
    assert np.array_equal(ref, got)
    with pytest.raises(ValueError):
        oracle.update(th, 0, s + [s[3]], np.append(q, 1), 1e-4, 9.0, 16.0)
    with pytest.raises(ValueError):
        oracle.canonical_order([(1, 2, 3), (1, 2, 3)])


def test_canonical_order_is_timestamp_order():
    seeds = [(5, 0, 1), (2, 9, 0), (5, 0, 0), (2, 1, 4), (9, 0, 0), (2, 1, 3)]
    perm = oracle.canonical_order(seeds)
    assert [seeds[i] for i in perm] == sorted(seeds)


def test_update_is_linear_in_pairs():
    idx = np.array([0, 1, 2, 3, 5, 1 << 33, (1 << 34) + 7], dtype=np.uint64)
    s = _seeds(4)
    q = np.array([3, -100, 127, -128], dtype=np.int8)
    whole = oracle.update_delta_at(idx, s, q, 1e-3, 4.0, 8.0)
    parts = sum(oracle.update_delta_at(idx, [s[k]], q[k:k + 1], 1e-3, 4.0, 8.0) for k in range(4))
    np.testing.assert_allclose(whole, parts, rtol=1e-14, atol=1e-20)
    # each part is c_k z_k
    for k in range(4):
        c = oracle.coefficient(q[k], 1e-3, 4.0, 8.0)
        np.testing.assert_allclose(oracle.update_delta_at(idx, [s[k]], q[k:k + 1], 1e-3, 4.0, 8.0),
                                   c * oracle.gaussian_at(s[k], idx), rtol=1e-15)


def test_update_delta_abs_is_delta_and_magnitude():
    """The one-pass (sum c z, sum |c z|) helper: its sum is update_delta_at's bit for
    bit, and update_at is the storage rounding of theta + that sum; its magnitude is
    sum_k |c_k| |z_k| term by term."""
    idx = np.array([0, 1, 2, 3, 5, 1 << 33, (1 << 34) + 7, 123456789], dtype=np.uint64)
    s = _seeds(6)
    q = np.array([3, -100, 127, -128, 0, 64], dtype=np.int8)
    delta, mag = oracle.update_delta_abs_at(idx, s, q, 1e-3, 6.0, 8.0)
    assert np.array_equal(delta, oracle.update_delta_at(idx, s, q, 1e-3, 6.0, 8.0))
    want = sum(abs(oracle.coefficient(q[k], 1e-3, 6.0, 8.0)) * np.abs(oracle.gaussian_at(s[k], idx))
               for k in range(6))
    np.testing.assert_allclose(mag, want, rtol=1e-14)
    assert np.all(mag >= np.abs(delta))
    th = oracle.round_bf16(synthetic.normal_values(idx.size, 0.02, 8).astype(np.float64))
    assert np.array_equal(oracle.update_at(th, idx, s, q, 1e-3, 6.0, 8.0),
                          oracle.round_bf16(oracle.bf16_to_f64(th) + delta))


def test_update_at_matches_contiguous():
    th = synthetic.normal_values(4096, 0.02, 6)
    hb = oracle.round_bf16(th.astype(np.float64))
    s = _seeds(5)
    q = synthetic.byte_codes(5, 2)
    for arr in (th, hb):
        full = oracle.update(arr, 100, s, q, 1e-3, 1.0, 16.0)
        idx = np.arange(100, 100 + arr.size, dtype=np.uint64)
        assert np.array_equal(oracle.update_at(arr, idx, s, q, 1e-3, 1.0, 16.0), full)
        assert np.array_equal(oracle.perturb_at(arr, idx, s[0], 0.5),
                              oracle.perturb(arr, 100, s[0], 0.5))


# --- SPSA estimator -----------------------------------------------------------

def test_spsa_quadratic_closed_form():
    """(L(theta + eps z) - L(theta - eps z)) / 2 eps = grad L . z for a quadratic."""
    toy = synthetic.toy_quadratic(1 << 16)
    th = toy.theta0.astype(np.float64)
    z = oracle.gaussian_range((1, 0, 0), 0, th.size)
    eps = 1e-3
    L = lambda t: 0.5 * np.sum(toy.a * (t - toy.target) ** 2)
    g_fd = (L(th + eps * z) - L(th - eps * z)) / (2 * eps)
    g_cf = np.dot(toy.a * (th - toy.target), z)
    assert abs(g_fd - g_cf) <= 1e-9 * np.sum(np.abs(toy.a * (th - toy.target) * z))


def test_spsa_unbiased_projected_gradient():
    """E[(g . z) z] = g with Var[(g . z) z_i] = |g|^2 + g_i^2, over 10^6 samples."""
    n, m = 16, 1_000_000
    g = synthetic.rng(4).standard_normal(n)
    acc = np.zeros(n)
    for j in range(m // 50_000):
        # 50,000 perturbation vectors of n parameters from one stream per chunk
        Z = oracle.gaussian_range((1234, j, 0), 0, 50_000 * n).reshape(50_000, n)
        acc += ((Z @ g)[:, None] * Z).sum(axis=0)
    est = acc / m
    se = np.sqrt((g @ g + g * g) / m)
    assert np.all(np.abs(est - g) < 5 * se)


def test_spsa_loop_descends_below_stability_limit():
    """Algorithm 1 on the quadratic: with eta / K below 2 / (n E[a]) the loss falls."""
    from oracle import spsa
    toy = synthetic.toy_quadratic(1 << 12)
    mids = synthetic.toy_machine_ids()
    L0 = spsa.quadratic_loss(toy.theta0, toy.a, toy.target)
    theta, recs = spsa.spsa_run(toy.theta0, toy.a, toy.target, mids, 8, 1e-3, 1e-3, 16.0)
    losses = [L0] + [r.loss_after for r in recs]
    assert losses[-1] < 0.995 * L0 and np.all(np.diff(losses) < 0)
    # each projected gradient equals grad L . z up to the fp32 storage of theta +- eps z
    r = recs[0]
    g = toy.a * (toy.theta0.astype(np.float64) - toy.target)
    for s, gh in zip(r.seeds, r.ghat):
        z = oracle.gaussian_range(s, 0, toy.theta0.size)
        assert abs(gh - g @ z) < 1e-3 * np.sum(np.abs(g * z))
    assert all(c == oracle.quantize(gh, 16.0) for c, gh in zip(r.codes, r.ghat))
