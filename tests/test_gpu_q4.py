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


SIZES = [1, 2, 31, 32, 33, 63, 64, 65, 96, 97, 127, 1000, 4097, 64 * 300 + 33]


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


def _check_codes(gc, want, w, scale_blocks, eps, mids):
    """Codes equal the oracle's except within fp32 error of a midpoint."""
    scale = np.repeat(scale_blocks.astype(np.float64), 64)[: w.size]
    x = np.where(scale > 0, w / np.where(scale > 0, scale, 1), 0.0)
    tol = (2e-6 * eps + 4e-7 * scale) / np.where(scale > 0, scale, 1) + 4e-7
    d = np.abs(x[:, None] - mids[None, :])
    near = d.min(axis=1) <= tol
    j = d.argmin(axis=1)
    return (gc == want) | (near & ((gc == j) | (gc == j + 1)))


def test_q4_perturb_zero_blocks(jb):
    """All-zero blocks: with eps = 0 they stay zero (scale 0, every code the zero
    level); with eps > 0 they take the noise alone."""
    sizes = [64 * 5 + 7, 130]
    offs = offsets(sizes)
    host, dev = [], []
    for i, n in enumerate(sizes):
        w = synthetic.normal_values(n, 0.02, 90 + i).astype(np.float64)
        w[64:192] = 0.0 if n > 192 else w[64:192]
        w[:64] = 0.0
        codes, scale = oracle.q4_quantize(w)
        host.append((codes, scale, n))
        pad = np.zeros(codes.size + 16, dtype=np.uint8)
        pad[: codes.size] = codes
        dev.append((torch.from_numpy(pad).cuda(), torch.from_numpy(scale.copy()).cuda(), n))
    table = jb.Q4Table(dev, offs)
    jb.jb_perturb_q4(table, (9, 9, 9), 0.0)
    torch.cuda.synchronize()
    zero_code = int(np.argmin(np.abs(oracle.q4_levels())))
    for (c, s, n), (dc, ds, _) in zip(host, dev):
        assert np.array_equal(dc.cpu().numpy()[: c.size], c)
        assert ds.cpu().numpy()[0] == 0.0
        assert np.all(codes_of(dc.cpu().numpy(), n)[:64] == zero_code)
    eps = float(F32(1e-3))
    seed = (77, 1, 2)
    jb.jb_perturb_q4(table, seed, eps)
    torch.cuda.synchronize()
    lev = oracle.q4_levels().astype(np.float64)
    mids = (lev[:-1] + lev[1:]) / 2
    for (c, s, n), (dc, ds, _), fo in zip(host, dev, offs):
        oc, os_, w = oracle.q4_perturb(c, s, n, fo, seed, eps)
        gs = ds.cpu().numpy()
        assert np.all(np.abs(gs.astype(np.float64) - os_) <= 2e-6 * os_ + 2e-6 * eps)
        ok = _check_codes(codes_of(dc.cpu().numpy(), n), codes_of(oc, n), w, os_, eps, mids)
        assert np.all(ok), (n, np.nonzero(~ok)[0][:5])


def test_q4_perturb_large_sampled(jb):
    """A multi-tensor set of 2^24+ elements with ragged sizes, checked on 3000
    random 64-element blocks, each block recomputed by the oracle on its own
    (a block depends only on its own codes, scale and global indices)."""
    sizes = [(1 << 23) + 64 * 3, 5_000_003, 64 * 37 + 1, (1 << 22) - 17]
    offs = offsets(sizes)
    host, dev, table = make(jb, sizes, offs, stream=95)
    seed = (0x1234_5678_9ABC, 3, 0)
    eps = float(F32(1e-2))
    jb.jb_perturb_q4(table, seed, eps)
    torch.cuda.synchronize()
    lev = oracle.q4_levels().astype(np.float64)
    mids = (lev[:-1] + lev[1:]) / 2
    rng = synthetic.rng(96)
    n_bad = 0
    for (c, s, n), (dc, ds, _), fo in zip(host, dev, offs):
        gcodes, gscale = dc.cpu().numpy(), ds.cpu().numpy()
        n_blocks = (n + 63) // 64
        for b in rng.choice(n_blocks, size=min(n_blocks, 750), replace=False):
            m = min(64, n - 64 * b)
            cb = c[32 * b: 32 * b + (m + 1) // 2]
            oc, os_, w = oracle.q4_perturb(cb, s[b: b + 1], m, fo + 64 * b, seed, eps)
            assert abs(float(gscale[b]) - float(os_[0])) <= 2e-6 * float(os_[0]) + 2e-6 * eps, (n, b)
            got = codes_of(gcodes[32 * b: 32 * b + (m + 1) // 2], m)
            ok = _check_codes(got, codes_of(oc, m), w, os_, eps, mids)
            n_bad += int(np.sum(~ok))
    assert n_bad == 0


def test_q4_perturb_full_size_13b_sampled(jb):
    """The OPT-13B-shaped set stored as 4-bit codes (12,853,473,280 elements in 644
    tensors, 6.4 GB of codes), perturbed in the launch the benchmark times; 4096
    random 64-element blocks, drawn over the whole set, each recomputed by the
    oracle from its codes and scale before the pass."""
    specs = synthetic.opt_tensors("opt-13b")
    g = torch.Generator(device="cuda")
    g.manual_seed(synthetic.MASTER_SEED + 41)
    tensors = []
    for sp in specs:
        n = sp.numel
        codes = torch.randint(0, 256, ((n + 1) // 2 + 8,), dtype=torch.uint8, device="cuda", generator=g)
        scale = torch.rand(((n + 63) // 64,), device="cuda", generator=g) * 0.05
        tensors.append((codes, scale, n))
    table = jb.Q4Table(tensors)
    n_blocks = np.array([(n + 63) // 64 for _, _, n in tensors], dtype=np.int64)
    first = np.concatenate([[0], np.cumsum(n_blocks)])
    pick = synthetic.rng(97).choice(int(first[-1]), size=4096, replace=False)
    which = np.searchsorted(first, pick, side="right") - 1
    ar = torch.arange(32, device="cuda")

    def gather():
        out = {}
        for t in np.unique(which):
            codes, scale, n = tensors[t]
            bl = torch.from_numpy(pick[which == t] - first[t]).cuda()
            idx = (32 * bl[:, None] + ar[None, :]).clamp_(max=codes.numel() - 1)
            out[int(t)] = (bl.cpu().numpy(), codes[idx].cpu().numpy(), scale[bl].cpu().numpy())
        return out

    before = gather()
    seed = (0x5EED_0013_B000, 11, 2)
    eps = float(F32(1e-3))
    jb.jb_perturb_q4(table, seed, eps)
    torch.cuda.synchronize()
    after = gather()
    lev = oracle.q4_levels().astype(np.float64)
    mids = (lev[:-1] + lev[1:]) / 2
    n_bad = n_checked = 0
    for t, (bl, c0, s0) in before.items():
        _, c1, s1 = after[t]
        n = tensors[t][2]
        fo = table.flat_offsets[t]
        for k, b in enumerate(bl):
            m = int(min(64, n - 64 * b))
            nb = (m + 1) // 2
            oc, os_, w = oracle.q4_perturb(c0[k, :nb].copy(), s0[k:k + 1], m, fo + 64 * int(b), seed, eps)
            assert abs(float(s1[k]) - float(os_[0])) <= 2e-6 * float(os_[0]) + 2e-6 * eps, (t, b)
            ok = _check_codes(codes_of(c1[k, :nb], m), codes_of(oc, m), w, os_, eps, mids)
            n_bad += int(np.sum(~ok))
            n_checked += m
    print(f"13B-shaped 4-bit set: {n_checked} elements in {len(pick)} blocks checked")
    assert n_bad == 0
    del tensors, table
    torch.cuda.empty_cache()
