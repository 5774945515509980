"""Parity of the CUDA path (through the C ABI) with the CPU oracle.

Bit-exact: the Philox stream (also against cuRAND's curand_Philox4x32_10) and
GPU-vs-GPU repeatability. Within tolerance: z (1e-6 absolute), fp32 theta
(2e-6 relative to the operands), bf16 theta (1 bf16 step). Sizes span many
warp tiles with ragged tails; edge cases cover empty and one-element tensors,
misaligned pointers, flat offsets whose phase defeats the vector path, and
Philox blocks above 2^32.
"""
import ctypes
import os
import subprocess

import numpy as np
import pytest

import oracle
import synthetic
from jbtest_util import (WIDENED, Z_ABS_TOL, as_f64, check_theta, to_device, to_host,
                         update_scale)

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
F32 = np.float32
LR, DENOM, QS = float(F32(1e-3)), float(F32(1.0)), 16.0


@pytest.fixture(scope="module")
def jb():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2306_10015_gb300 import build
    build.build()
    import paper_2306_10015_gb300 as pkg
    pkg.lib()
    return pkg


def sync():
    torch.cuda.synchronize()


# --- the random stream ----------------------------------------------------------

SEEDS = [(0, 0, 0), (0xFFFFFFFFFFFFFFFF, 0xFFFFFFFF, 0xFFFFFFFF), (1_700_000_000_000_000_137, 3, 0),
         (0xDEADBEEF00000000, 12345, 77)]


@pytest.mark.parametrize("seed", SEEDS)
def test_philox_stream_bit_exact(jb, seed):
    for first in (0, (1 << 32) - 1000, 7_493_600_000):
        n = 1 << 16
        out = torch.empty(4 * n, dtype=torch.int32, device="cuda")
        jb.jb_debug_philox(seed, first, n, out)
        sync()
        got = out.cpu().numpy().view(np.uint32).reshape(n, 4)
        assert np.array_equal(got, oracle.philox_blocks(seed, first, n))


@pytest.mark.parametrize("seed", SEEDS[:3])
def test_philox_fold_bit_exact(jb, seed):
    """The generator-only kernel (the benchmark's generator floor) folds exactly the
    words the oracle draws, on ragged counts and across the 2^32-block boundary."""
    out = torch.zeros(1, dtype=torch.int32, device="cuda")
    for first, n in ((0, 1 << 20), ((1 << 32) - 5000, 77_777), (7_493_600_000, 1), (12, 0)):
        jb.jb_debug_philox_fold(seed, first, n, out)
        sync()
        got = int(out.cpu().numpy().view(np.uint32)[0])
        want = int(np.bitwise_xor.reduce(oracle.philox_blocks(seed, first, n).ravel())) if n else 0
        assert got == want, (first, n)


@pytest.fixture(scope="module")
def curand_lib():
    src = os.path.join(ROOT, "tests", "helpers", "curand_philox.cu")
    out_dir = os.path.join(ROOT, "tests", "_build")
    os.makedirs(out_dir, exist_ok=True)
    so = os.path.join(out_dir, "libcurand_philox.so")
    if not os.path.exists(so) or os.path.getmtime(src) > os.path.getmtime(so):
        subprocess.run(["nvcc", "-gencode", "arch=compute_103a,code=sm_103a", "-O2", "-shared",
                        "-Xcompiler", "-fPIC", src, "-o", so], check=True)
    L = ctypes.CDLL(so)
    L.curand_philox_blocks.argtypes = [ctypes.c_void_p] * 3 + [ctypes.c_uint64]
    return L


def test_philox_matches_curand(jb, curand_lib):
    n = 1 << 15
    g = synthetic.rng(11)
    mids = g.integers(0, 2**64, size=n, dtype=np.uint64)
    steps = g.integers(0, 2**32, size=n, dtype=np.uint64).astype(np.uint32)
    samples = g.integers(0, 2**32, size=n, dtype=np.uint64).astype(np.uint32)
    blocks = g.integers(0, 2**40, size=n, dtype=np.uint64)
    ctr = np.stack([blocks & 0xFFFFFFFF, blocks >> 32, steps, samples], 1).astype(np.uint32)
    key = np.stack([mids & 0xFFFFFFFF, mids >> 32], 1).astype(np.uint32)
    d_ctr = torch.from_numpy(ctr.view(np.int32)).cuda()
    d_key = torch.from_numpy(key.view(np.int32)).cuda()
    d_out = torch.empty((n, 4), dtype=torch.int32, device="cuda")
    assert curand_lib.curand_philox_blocks(d_ctr.data_ptr(), d_key.data_ptr(), d_out.data_ptr(), n) == 0
    ref = d_out.cpu().numpy().view(np.uint32)
    mine = torch.empty(4, dtype=torch.int32, device="cuda")
    for i in range(0, n, 2048):  # library hook, one block at a time per distinct seed
        jb.jb_debug_philox((int(mids[i]), int(steps[i]), int(samples[i])), int(blocks[i]), 1, mine)
        sync()
        assert np.array_equal(mine.cpu().numpy().view(np.uint32), ref[i])


def test_gaussian_parity_1e8(jb):
    """|z_gpu - z| <= 1e-6 over 10^8 draws from several seeds."""
    worst = 0.0
    chunk = 1 << 24
    buf = torch.empty(chunk, dtype=torch.float32, device="cuda")
    drawn = 0
    for i, seed in enumerate([(synthetic.MASTER_SEED + i, i, 3 * i) for i in range(6)]):
        first = i * 1_000_003 + (0 if i % 2 else (1 << 34) - chunk // 2)
        jb.jb_debug_gaussian(seed, first, chunk, buf)
        sync()
        got = buf.cpu().numpy().astype(np.float64)
        want = oracle.gaussian_range(seed, first, chunk)
        worst = max(worst, float(np.max(np.abs(got - want))))
        drawn += chunk
    assert drawn >= 10**8
    print(f"max |dz| over {drawn} draws: {worst:.3e}")
    assert worst <= Z_ABS_TOL


def test_box_muller_extremes(jb):
    """Every radius word at two angles, every angle word at the largest radius, and the
    largest radii (u_a -> 0) with the angles nearest the axes."""
    ma = np.arange(0, 1 << 12, dtype=np.uint32)
    angles = np.concatenate([np.arange(0, 64, dtype=np.uint32),
                             (np.arange(4, dtype=np.uint32) << 22)[:, None].ravel(),
                             synthetic.rng(12).integers(0, 1 << 24, 200).astype(np.uint32)])
    xa = np.repeat(ma << 9, angles.size)
    xb = np.tile(angles << 8, ma.size)
    all_b = np.arange(0, 1 << 24, dtype=np.uint32) << 8
    all_a = np.arange(0, 1 << 23, dtype=np.uint32) << 9
    xa = np.concatenate([xa, np.zeros(all_b.size, np.uint32), np.full(4096, 0xFFFFFFFF, np.uint32),
                         all_a, all_a])
    # every radius word at the angle nearest 0 (cos ~ 1) and nearest pi/4 (|cos| = |sin|)
    xb = np.concatenate([xb, all_b, np.arange(4096, dtype=np.uint32) << 12,
                         np.zeros(all_a.size, np.uint32), np.full(all_a.size, 0x1FFFFF << 8, np.uint32)])
    words = np.stack([xa, xb], 1).reshape(-1)
    n = xa.size
    d_words = torch.from_numpy(words.view(np.int32)).cuda()
    out = torch.empty(2 * n, dtype=torch.float32, device="cuda")
    jb.jb_debug_box_muller(d_words, n, out)
    sync()
    got = out.cpu().numpy().astype(np.float64).reshape(n, 2)
    want = oracle.box_muller_pairs(words.reshape(n, 2))
    err = np.abs(got - want)
    rel = err / np.maximum(np.abs(want), 1e-30)
    print(f"max |dz| over all radius words and all angle words: {err.max():.3e}, "
          f"max relative {rel.max():.3e}")
    assert err.max() <= Z_ABS_TOL
    # relative accuracy of the small members (the zeros of cos and sin are exact in angle)
    small = np.abs(want) < 1e-3
    assert np.all(err[small] <= 4 * np.spacing(np.abs(want[small]).astype(np.float32)))


def test_box_muller_joint_worst(jb):
    """The radius and the angle are computed independently, so the worst |dz| pairs
    a large radius error with a large angle error. The radius of every radius word
    is read at angle word 0 (the cosine is then exactly 1, z = r); the 64 words whose
    radius is furthest from sqrt(-2 ln u_a) in double precision, and the 32 largest
    radii (where an angle error weighs most), are each taken with all 2^24 angle
    words (1.6e9 draws) against the oracle."""
    all_a = np.arange(0, 1 << 23, dtype=np.uint32) << 9
    words = np.stack([all_a, np.zeros_like(all_a)], 1).reshape(-1)
    out = torch.empty(words.size, dtype=torch.float32, device="cuda")
    jb.jb_debug_box_muller(torch.from_numpy(words.view(np.int32)).cuda(), all_a.size, out)
    sync()
    r_gpu = out.cpu().numpy().astype(np.float64)[0::2]
    u_a = ((all_a >> 9).astype(np.float64) + 0.5) * 2.0**-23
    dr = np.abs(r_gpu - np.sqrt(-2.0 * np.log(u_a)))
    worst = np.union1d(np.argsort(dr)[-64:], np.arange(32))  # word 0: the largest radius
    all_b = np.arange(0, 1 << 24, dtype=np.uint32) << 8
    out = torch.empty(2 * all_b.size, dtype=torch.float32, device="cuda")
    m = 0.0
    for k in worst:
        pairs = np.stack([np.full(all_b.size, all_a[k], np.uint32), all_b], 1)
        jb.jb_debug_box_muller(torch.from_numpy(pairs.reshape(-1).view(np.int32)).cuda(),
                               all_b.size, out)
        sync()
        got = out.cpu().numpy().astype(np.float64).reshape(-1, 2)
        m = max(m, float(np.abs(got - oracle.box_muller_pairs(pairs)).max()))
    print(f"largest radius error {dr.max():.3e}; max |dz| over {worst.size} radius words "
          f"x every angle word: {m:.3e}")
    assert m <= Z_ABS_TOL


# --- layouts --------------------------------------------------------------------

def make_layout(kind: str, dtype):
    """(host arrays, flat offsets, pointer offsets in elements) for a test layout."""
    if kind == "ragged":
        sizes = synthetic.ragged_sizes(37, 70_000, 1)
        offs = synthetic.flat_offsets(sizes)
        shifts = [0] * len(sizes)
    elif kind == "phase":
        # flat offsets not multiple of the vector width, and tensors that start 1 or 3
        # elements past a 16-byte boundary: some take the vector path, some do not
        sizes = synthetic.ragged_sizes(23, 40_000, 2)
        offs, cur = [], 5
        for i, n in enumerate(sizes):
            offs.append(cur)
            cur += n + (i % 5)
        shifts = [(i * 3) % 8 for i in range(len(sizes))]
    elif kind == "tiny":
        sizes = list(range(1, 34))
        offs, cur = [], 0
        for n in sizes:
            offs.append(cur)
            cur += n + 1
        shifts = [i % 4 for i in range(len(sizes))]
    elif kind == "high":
        # global indices above 2^34: Philox block indices above 2^32, with a crossing
        sizes = [1000, 4097, 333, 65536]
        offs = [(1 << 34) - 2000, (1 << 34) - 1000 + 8, 1 << 36, (1 << 40) + 3]
        shifts = [0, 0, 1, 0]
    else:
        raise ValueError(kind)
    vals = []
    for i, n in enumerate(sizes):
        v = synthetic.normal_values(n, 0.02, 50 + i)
        if i % 6 == 5:
            v[:] = 0.0  # zero biases
        if i % 6 == 4:
            v[:] = 1.0  # LayerNorm gains
        vals.append(v if dtype == "f32" else oracle.round_bf16(v.astype(np.float64)))
    return vals, offs, shifts


def upload(jb, vals, offs, shifts):
    """Tensors at the requested element shifts inside a padded allocation."""
    tensors, keep = [], []
    for v, sh in zip(vals, shifts):
        pad = np.zeros(v.size + 16, dtype=v.dtype)
        base = to_device(pad)
        t = base[sh:sh + v.size]
        t.copy_(to_device(v))
        tensors.append(t)
        keep.append(base)
    table = jb.ParamTable(tensors, offs)
    table._keep = keep
    return table


def download(table):
    return [to_host(t) for t in table.tensors]


LAYOUTS = ["ragged", "phase", "tiny", "high"]


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
@pytest.mark.parametrize("kind", LAYOUTS)
def test_perturb_parity(jb, dtype, kind):
    vals, offs, shifts = make_layout(kind, dtype)
    table = upload(jb, vals, offs, shifts)
    seed, eps = (0x1234_5678_9ABC_DEF0, 7, 2), float(F32(1e-3))
    jb.jb_perturb(table, seed, eps)
    sync()
    worst, mark = 0.0, len(WIDENED)
    for v, fo, got in zip(vals, offs, download(table)):
        want = oracle.perturb(v, fo, seed, eps)
        z = oracle.gaussian_range(seed, fo, v.size)
        worst = max(worst, check_theta(got, want, np.abs(as_f64(v)) + eps * np.abs(z), kind))
    print(f"{kind}/{dtype}: worst error / allowance = {worst:.3f}; {_widened(mark)}")


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_perturb_restore_cycle(jb, dtype):
    """+eps, -2 eps, +eps (Algorithm 1) restores theta up to three roundings."""
    vals, offs, shifts = make_layout("ragged", dtype)
    table = upload(jb, vals, offs, shifts)
    seed, eps = (99, 1, 0), float(F32(1e-3))
    for e in (eps, -2 * eps, eps):
        jb.jb_perturb(table, seed, e)
    sync()
    for v, fo, got in zip(vals, offs, download(table)):
        z = np.abs(oracle.gaussian_range(seed, fo, v.size))
        scale = np.abs(as_f64(v)) + 2 * eps * z
        if dtype == "f32":
            ulp = np.spacing(scale.astype(np.float32)).astype(np.float64)
        else:
            ulp = np.ldexp(1.0, np.frexp(scale)[1] - 8)
        assert np.all(np.abs(as_f64(got) - as_f64(v)) <= 1.5 * ulp + 1e-40)


def _widened(mark: int) -> str:
    """Elements beyond one bf16 step (admitted by the fp32 allowance) since WIDENED[mark]."""
    n = sum(w for _, w, _ in WIDENED[mark:])
    tot = sum(t for _, _, t in WIDENED[mark:])
    return f"{n} of {tot} elements beyond one bf16 step" if tot else "fp32"


def _pairs(K, step=3, stream=0):
    mids = synthetic.machine_ids(K, 20 + stream)
    seeds = [(int(m), step, int(i % 3)) for i, m in enumerate(mids)]
    q = synthetic.byte_codes(K, 20 + stream)
    return seeds, q


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
@pytest.mark.parametrize("K", [1, 2, 3, 17, 64])
@pytest.mark.parametrize("kind", ["ragged", "phase", "high", "tiny"])
def test_update_parity(jb, dtype, K, kind):
    vals, offs, shifts = make_layout(kind, dtype)
    table = upload(jb, vals, offs, shifts)
    seeds, q = _pairs(K)
    jb.jb_apply_updates(table, seeds, q, LR, DENOM, QS)
    sync()
    worst, mark = 0.0, len(WIDENED)
    for v, fo, got in zip(vals, offs, download(table)):
        want = oracle.update(v, fo, seeds, q, LR, DENOM, QS)
        idx = np.arange(fo, fo + v.size, dtype=np.uint64)
        scale = update_scale(v, idx, seeds, q, LR, DENOM, QS)
        worst = max(worst, check_theta(got, want, scale, f"{kind} K={K}"))
    print(f"{kind}/{dtype}/K={K}: worst error / allowance = {worst:.3f}; {_widened(mark)}")


def test_update_k256_parity(jb):
    vals, offs, shifts = make_layout("ragged", "f32")
    vals, offs, shifts = vals[:6], offs[:6], shifts[:6]
    table = upload(jb, vals, offs, shifts)
    seeds, q = _pairs(256, stream=5)
    jb.jb_apply_updates(table, seeds, q, LR, float(F32(256.0)), QS)
    sync()
    for v, fo, got in zip(vals, offs, download(table)):
        want = oracle.update(v, fo, seeds, q, LR, 256.0, QS)
        idx = np.arange(fo, fo + v.size, dtype=np.uint64)
        check_theta(got, want, update_scale(v, idx, seeds, q, LR, 256.0, QS), "K=256")


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_update_max_pairs_parity(jb, dtype):
    """K = jb_max_seeds_per_call() (512): the largest list one launch carries."""
    K = jb.jb_max_seeds_per_call()
    vals, offs, shifts = make_layout("phase", dtype)
    vals, offs, shifts = vals[:5], offs[:5], shifts[:5]
    table = upload(jb, vals, offs, shifts)
    seeds, q = _pairs(K, stream=6)
    jb.jb_apply_updates(table, seeds, q, LR, float(F32(K)), QS)
    sync()
    mark = len(WIDENED)
    for v, fo, got in zip(vals, offs, download(table)):
        want = oracle.update(v, fo, seeds, q, LR, float(K), QS)
        idx = np.arange(fo, fo + v.size, dtype=np.uint64)
        check_theta(got, want, update_scale(v, idx, seeds, q, LR, float(K), QS), f"K={K}")
    print(f"K={K}/{dtype}: {_widened(mark)}")


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_update_k1_matches_perturb(jb, dtype):
    vals, offs, shifts = make_layout("ragged", dtype)
    a = upload(jb, vals, offs, shifts)
    b = upload(jb, vals, offs, shifts)
    seeds, q = _pairs(1)
    jb.jb_apply_updates(a, seeds, q, LR, DENOM, QS)
    jb.jb_perturb(b, seeds[0], oracle.coefficient(int(q[0]), LR, DENOM, QS))
    sync()
    for v, fo, x, y in zip(vals, offs, download(a), download(b)):
        scale = np.abs(as_f64(v)) + abs(oracle.coefficient(int(q[0]), LR, DENOM, QS)) * np.abs(
            oracle.gaussian_range(seeds[0], fo, v.size))
        check_theta(x, y, scale, "K=1 vs perturb")


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_update_order_invariance_bitwise(jb, dtype):
    vals, offs, shifts = make_layout("ragged", dtype)
    seeds, q = _pairs(40)
    perm = synthetic.rng(13).permutation(40)
    outs = []
    for order in (np.arange(40), perm):
        t = upload(jb, vals, offs, shifts)
        jb.jb_apply_updates(t, [seeds[i] for i in order], q[order], LR, DENOM, QS)
        sync()
        outs.append(download(t))
    for x, y in zip(*outs):
        assert np.array_equal(x, y)


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_repeatable_across_runs_grids_and_splits(jb, dtype):
    """Bitwise identical results for any grid and any split of the same indices."""
    n, fo = 300_001, 1 << 20
    v = synthetic.normal_values(n, 0.02, 90)
    v = v if dtype == "f32" else oracle.round_bf16(v.astype(np.float64))
    seeds, q = _pairs(9)
    one_s, one_q = _pairs(1, stream=4)  # K = 1 takes the one-pair kernel
    ref = None
    for grid in (0, 0, 1, 7, 152, 1000):
        t = upload(jb, [v], [fo], [0])
        jb.jb_apply_updates(t, seeds, q, LR, DENOM, QS, grid_ctas=grid)
        jb.jb_perturb(t, seeds[0], 1e-3, grid_ctas=grid)
        jb.jb_apply_updates(t, one_s, one_q, LR, DENOM, QS, grid_ctas=grid)
        sync()
        out = download(t)[0]
        if ref is None:
            ref = out
        assert np.array_equal(out, ref), grid
    cuts = [0, 1, 17, 4096, 4097, 100_000, 299_999, n]
    parts = [v[a:b] for a, b in zip(cuts[:-1], cuts[1:])]
    t = upload(jb, parts, [fo + a for a in cuts[:-1]], [(i * 5) % 8 for i in range(len(parts))])
    jb.jb_apply_updates(t, seeds, q, LR, DENOM, QS)
    jb.jb_perturb(t, seeds[0], 1e-3)
    jb.jb_apply_updates(t, one_s, one_q, LR, DENOM, QS)
    sync()
    assert np.array_equal(np.concatenate(download(t)), ref)


def test_zero_eps_and_empty_segments(jb):
    vals, offs, shifts = make_layout("tiny", "bf16")
    table = upload(jb, vals, offs, shifts)
    jb.jb_perturb(table, (5, 5, 5), 0.0)
    jb.jb_apply_updates(table, [], [], LR, DENOM, QS)
    sync()
    for v, got in zip(vals, download(table)):
        assert np.array_equal(v, got)
    # zero-length tensors in the table are skipped
    empty = torch.empty(0, dtype=torch.bfloat16, device="cuda")
    t = jb.ParamTable([empty, table.tensors[3]], [0, offs[3]])
    jb.jb_perturb(t, (5, 5, 5), 1e-3)
    sync()
    assert np.array_equal(to_host(t.tensors[1]), oracle.perturb(vals[3], offs[3], (5, 5, 5),
                                                                float(F32(1e-3))))


def test_side_stream(jb):
    vals, offs, shifts = make_layout("ragged", "f32")
    table = upload(jb, vals, offs, shifts)
    s = torch.cuda.Stream()
    seeds, q = _pairs(4)
    with torch.cuda.stream(s):
        jb.jb_apply_updates(table, seeds, q, LR, DENOM, QS, stream=s)
    s.synchronize()
    for v, fo, got in zip(vals, offs, download(table)):
        idx = np.arange(fo, fo + v.size, dtype=np.uint64)
        check_theta(got, oracle.update(v, fo, seeds, q, LR, DENOM, QS),
                    update_scale(v, idx, seeds, q, LR, DENOM, QS), "side stream")


def test_many_segments_split_across_launches(jb):
    """More tensors than one launch's parameter space holds (the 30B-shaped set has 772)."""
    sizes = [int(s) for s in synthetic.ragged_sizes(1500, 300, 3)]
    offs = synthetic.flat_offsets(sizes)
    vals = [oracle.round_bf16(synthetic.normal_values(n, 0.02, 3000 + i).astype(np.float64))
            for i, n in enumerate(sizes)]
    flat = np.concatenate(vals)
    big = to_device(np.concatenate([flat, np.zeros(8, np.uint16)]))
    tensors, cur = [], 0
    for n in sizes:
        tensors.append(big[cur:cur + n])
        cur += n
    table = jb.ParamTable(tensors, offs)
    seeds, q = _pairs(5)
    jb.jb_apply_updates(table, seeds, q, LR, DENOM, QS)
    jb.jb_perturb(table, seeds[1], 1e-3)
    sync()
    got = to_host(big[:flat.size])
    idx = np.concatenate([np.arange(fo, fo + n, dtype=np.uint64) for fo, n in zip(offs, sizes)])
    mid = oracle.update_at(flat, idx, seeds, q, LR, DENOM, QS)
    want = oracle.perturb_at(mid, idx, seeds[1], float(F32(1e-3)))
    d = np.abs(np.where(got & 0x8000, -(got & 0x7FFF).astype(np.int64), got.astype(np.int64)) -
               np.where(want & 0x8000, -(want & 0x7FFF).astype(np.int64), want.astype(np.int64)))
    assert d.max() <= 2  # two bf16 roundings on each side
