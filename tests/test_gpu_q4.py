"""PerturbParameters on 4-bit weights (Section 3) against the oracle.

The code of an element is an integer decided in floating point: it must equal
the oracle's, except where the oracle's w'/scale' lies within the fp32 error of
a midpoint between two levels; there either neighbour is accepted."""
import numpy as np
import pytest

import oracle
import synthetic

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

F32 = np.float32


@pytest.fixture(scope="module")
def jb():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2306_10015_gb300 import build
    build.build()
    import paper_2306_10015_gb300 as pkg
    pkg.lib()
    return pkg


SIZES = [1, 2, 63, 64, 65, 127, 1000, 4097, 64 * 300 + 33]


def make(jb, sizes, offs, stream=70):
    host, dev = [], []
    for i, n in enumerate(sizes):
        w = synthetic.normal_values(n, 0.02, stream + i).astype(np.float64)
        codes, scale = oracle.q4_quantize(w)
        host.append((codes, scale, n))
        pad = np.zeros(codes.size + 16, dtype=np.uint8)
        pad[: codes.size] = codes
        dev.append((torch.from_numpy(pad).cuda(), torch.from_numpy(scale.copy()).cuda(), n))
    return host, dev, jb.Q4Table(dev, offs)


def codes_of(c, n):
    out = np.empty(n, dtype=np.int64)
    out[0::2] = c[: (n + 1) // 2] & 0xF
    out[1::2] = c[: n // 2] >> 4
    return out


def offsets(sizes):
    offs, cur = [], 4
    for n in sizes:
        offs.append(cur)
        cur = (cur + n + 3) // 4 * 4 + 4 * (len(offs) % 3)
    return offs


def test_zero_eps_is_identity(jb):
    host, dev, table = make(jb, SIZES, offsets(SIZES))
    jb.jb_perturb_q4(table, (1, 2, 3), 0.0)
    torch.cuda.synchronize()
    for (c, s, n), (dc, ds, _) in zip(host, dev):
        assert np.array_equal(dc.cpu().numpy()[: c.size], c)
        assert np.array_equal(ds.cpu().numpy(), s)


@pytest.mark.parametrize("eps", [1e-3, 2e-2])
def test_q4_perturb_parity(jb, eps):
    eps = float(F32(eps))
    offs = offsets(SIZES)
    host, dev, table = make(jb, SIZES, offs)
    seed = (0xABCDEF0123, 5, 1)
    jb.jb_perturb_q4(table, seed, eps)
    torch.cuda.synchronize()
    lev = oracle.q4_levels().astype(np.float64)
    mids = (lev[:-1] + lev[1:]) / 2
    near_total = 0
    for (c, s, n), (dc, ds, _), fo in zip(host, dev, offs):
        oc, os_, w = oracle.q4_perturb(c, s, n, fo, seed, eps)
        gs = ds.cpu().numpy()
        # scales: the largest |w'| of the block, fp32 error of the operands allowed
        assert np.all(np.abs(gs.astype(np.float64) - os_) <= 2e-6 * os_ + 2e-6 * eps), (n, fo)
        gc = codes_of(dc.cpu().numpy(), n)
        want = codes_of(oc, n)
        scale = np.repeat(os_.astype(np.float64), 64)[:n]
        x = np.where(scale > 0, w / np.where(scale > 0, scale, 1), 0.0)
        tol = (2e-6 * eps + 4e-7 * scale) / np.where(scale > 0, scale, 1) + 4e-7
        d = np.abs(x[:, None] - mids[None, :])
        near = d.min(axis=1) <= tol
        j = d.argmin(axis=1)
        ok = (gc == want) | (near & ((gc == j) | (gc == j + 1)))
        assert np.all(ok), (n, fo, np.nonzero(~ok)[0][:5])
        near_total += int(np.sum(near & (gc != want)))
        if n % 2 == 1:  # the unused high nibble of an odd tail is left as it was
            assert dc.cpu().numpy()[n // 2] >> 4 == c[n // 2] >> 4
    print(f"eps={eps}: codes decided differently within tolerance of a midpoint: {near_total}")
