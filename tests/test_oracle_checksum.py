"""Pins of the oracle's model checksum (ChecksumMatch, Algorithm 1)."""
import numpy as np
import pytest

import oracle
import synthetic

C0, C1 = 0x6A09E667, 0xF3BCC908


def aten_four_rounds(lib, words, k0, k1):
    out = np.empty(4, dtype=np.uint32)
    w = [int(x) for x in words]
    lib.aten_philox_rounds((k1 << 32) | k0, (w[3] << 32) | w[2], (w[1] << 32) | w[0], 4,
                           out.ctypes.data)
    return out


def test_window_hash_is_four_philox_rounds(aten_philox):
    g = synthetic.rng(40)
    for _ in range(500):
        v = int(g.integers(0, 2**62))
        words = g.integers(0, 2**32, size=4, dtype=np.uint64)
        x = aten_four_rounds(aten_philox, words, (v & 0xFFFFFFFF) ^ C0, (v >> 32) ^ C1)
        want = ((int(x[1]) << 32 | int(x[0])) + (int(x[3]) << 32 | int(x[2]))) % (1 << 64)
        assert oracle.window_hash(v, words) == want


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_checksum_sees_every_bit(dtype):
    v = synthetic.normal_values(200, 0.02, 41)
    a = v if dtype == "f32" else oracle.round_bf16(v.astype(np.float64))
    base = oracle.checksum([a], [13])
    bits = 32 if dtype == "f32" else 16
    seen = {base}
    for i in range(a.size):
        for b in range(bits):
            m = a.copy()
            m.view(np.uint32 if dtype == "f32" else np.uint16)[i] ^= (1 << b)
            h = oracle.checksum([m], [13])
            assert h != base
            seen.add(h)
    assert len(seen) == 1 + a.size * bits  # no two single-bit changes collide either


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_checksum_layout_invariances(dtype):
    E = 4 if dtype == "f32" else 8
    n = 1000 * E
    v = synthetic.normal_values(n, 0.02, 42)
    a = v if dtype == "f32" else oracle.round_bf16(v.astype(np.float64))
    whole = oracle.checksum([a], [E * 7])
    # splitting at window boundaries and listing the pieces in any order changes nothing
    cuts = [0, 3 * E, 100 * E, 101 * E, 640 * E, n]
    pieces = [(a[x:y], E * 7 + x) for x, y in zip(cuts[:-1], cuts[1:])]
    perm = [3, 0, 4, 2, 1]
    assert oracle.checksum([pieces[i][0] for i in perm], [pieces[i][1] for i in perm]) == whole
    # a partial window reads the missing elements as zero
    part = a[: 10 * E + 3]
    padded = np.concatenate([part, np.zeros(E - 3, dtype=a.dtype)])
    assert oracle.checksum([part], [E * 7]) == oracle.checksum([padded], [E * 7])
    # the checksum depends on where the values sit in the global index space
    assert oracle.checksum([a], [E * 8]) != whole
