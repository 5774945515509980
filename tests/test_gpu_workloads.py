"""Parity at the workloads' full sizes, through the C ABI in the launch
configuration the benchmark times, on sampled outputs the oracle computes one
by one; plus the toy SPSA run (Algorithm 1 end to end) and the dynamic-
membership run, both free-running against the oracle from the same inputs.

Inputs come from the seeded generators in `synthetic` (torch's generator on the
device for the OPT-shaped sets); the oracle never takes a value produced by the
CUDA path as input.
"""
import gc

import numpy as np
import pytest

import oracle
import synthetic
from jbtest_util import (WIDENED, as_f64, bf16_ord, check_theta, to_device, to_host,
                         update_scale)

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


def free_cuda():
    gc.collect()
    torch.cuda.synchronize()
    torch.cuda.empty_cache()


def gather(tensors, positions):
    parts = []
    for t, p in zip(tensors, positions):
        parts.append(to_host(t[torch.from_numpy(p).to(t.device)]))
    return np.concatenate(parts)


def global_index(offsets, positions):
    return np.concatenate([fo + p for fo, p in zip(offsets, positions)]).astype(np.uint64)


WORKLOADS = [("opt-125m", "f32", 16), ("opt-1.3b", "bf16", 64), ("opt-13b", "bf16", 64)]


def _setup(jb, model, dtype, n_samples=1 << 18):
    tdt = torch.float32 if dtype == "f32" else torch.bfloat16
    specs, tensors, offs = synthetic.opt_parameters(model, tdt)
    table = jb.ParamTable(tensors, offs)
    pos = synthetic.sample_positions([t.numel() for t in tensors], n_samples, 7)
    return table, pos, offs


@pytest.mark.parametrize("model,dtype,K", WORKLOADS)
def test_full_size_perturb_sampled(jb, model, dtype, K):
    table, pos, offs = _setup(jb, model, dtype)
    idx = global_index(offs, pos)
    before = gather(table.tensors, pos)
    seed, eps = (int(synthetic.machine_ids(1, 60)[0]), 11, 0), float(F32(1e-3))
    jb.jb_perturb(table, seed, eps)
    torch.cuda.synchronize()
    after = gather(table.tensors, pos)
    want = oracle.perturb_at(before, idx, seed, eps)
    scale = np.abs(as_f64(before)) + eps * np.abs(oracle.gaussian_at(seed, idx))
    worst = check_theta(after, want, scale, f"{model} perturb")
    print(f"{model}: {idx.size} sampled elements, worst error / allowance {worst:.3f}")
    del table
    free_cuda()


# the benchmark's K sweep ends: K = 1 runs the one-pair kernel, K = 256 the seed loop
UPDATE_WORKLOADS = WORKLOADS + [("opt-13b", "bf16", 1), ("opt-13b", "bf16", 256)]


@pytest.mark.parametrize("model,dtype,K", UPDATE_WORKLOADS)
def test_full_size_update_sampled(jb, model, dtype, K):
    table, pos, offs = _setup(jb, model, dtype)
    idx = global_index(offs, pos)
    before = gather(table.tensors, pos)
    seeds = [(int(m), 11, 0) for m in synthetic.machine_ids(K, 61)]
    q = synthetic.byte_codes(K, 61)
    lr, denom, qs = float(F32(1e-6)), 1.0, 16.0
    jb.jb_apply_updates(table, seeds, q, lr, denom, qs)
    torch.cuda.synchronize()
    after = gather(table.tensors, pos)
    want = oracle.update_at(before, idx, seeds, q, lr, denom, qs)
    worst = check_theta(after, want, update_scale(before, idx, seeds, q, lr, denom, qs),
                        f"{model} update K={K}")
    print(f"{model}: K={K}, {idx.size} sampled elements, worst error / allowance {worst:.3f}")
    del table
    free_cuda()


@pytest.mark.parametrize("K,write_src", [(1, False), (4, True)])
def test_full_size_apply_from_sampled_13b(jb, K, write_src):
    """The update read from the weight backup (Algorithm 1's restore fused) on the
    13B-shaped bf16 set, in the launches the benchmark times: K = 1 runs the
    one-pair kernel, K = 4 the grouped kernel with the backup refreshed."""
    backup, pos, offs = _setup(jb, "opt-13b", "bf16")
    theta = jb.ParamTable([torch.empty_like(t) for t in backup.tensors], offs)
    idx = global_index(offs, pos)
    before = gather(backup.tensors, pos)
    seeds = [(int(m), 9, 0) for m in synthetic.machine_ids(K, 920)]
    q = synthetic.byte_codes(K, 920)
    lr, denom, qs = float(F32(1e-6)), 1.0, 16.0
    jb.jb_apply_updates_from(backup, theta, seeds, q, lr, denom, qs, write_src=write_src)
    torch.cuda.synchronize()
    got = gather(theta.tensors, pos)
    src = gather(backup.tensors, pos)
    want = oracle.update_at(before, idx, seeds, q, lr, denom, qs)
    worst = check_theta(got, want, update_scale(before, idx, seeds, q, lr, denom, qs),
                        f"13B update from backup K={K}")
    assert np.array_equal(src, got if write_src else before)
    print(f"opt-13b from backup: K={K}, {idx.size} sampled elements, worst error / allowance {worst:.3f}")
    del backup, theta
    free_cuda()


def test_full_size_replay_sampled_13b(jb):
    """A late joiner's replay (Appendix B) of 16 steps x 4 pairs on the 13B-shaped
    bf16 set, each step rounded to storage as its own update would be: against the
    oracle stepping the sampled elements one update at a time."""
    table, pos, offs = _setup(jb, "opt-13b", "bf16")
    idx = global_index(offs, pos)
    want = gather(table.tensors, pos)
    lr, qs = float(F32(1e-6)), 16.0
    steps = []
    for t in range(16):
        seeds = [(int(m), 100 + t, 0) for m in synthetic.machine_ids(4, 930, t)]
        steps.append((seeds, synthetic.byte_codes(4, 930, t), lr, 4.0))
    jb.jb_replay_updates(table, [(jb.seeds_array(s), q, l, d) for s, q, l, d in steps], qs)
    torch.cuda.synchronize()
    got = gather(table.tensors, pos)
    allow = np.zeros(idx.size)
    for seeds, q, l, d in steps:
        scale = update_scale(want, idx, seeds, q, l, d, qs)
        allow += np.ldexp(1.0, np.frexp(scale)[1] - 8) + 2e-6 * scale
        want = oracle.update_at(want, idx, seeds, q, l, d, qs)
    err = np.abs(as_f64(got) - as_f64(want))
    ratio = float((err / (allow + 1e-300)).max())
    print(f"opt-13b replay 16 x 4: {idx.size} sampled elements, worst error / allowance {ratio:.3f}")
    assert np.all(err <= allow + 2.0**-133), ratio
    del table
    free_cuda()


def test_full_size_restore_cycle_13b(jb):
    """+eps, -2 eps, +eps on the 13B-shaped bf16 set: back within three roundings."""
    table, pos, offs = _setup(jb, "opt-13b", "bf16")
    idx = global_index(offs, pos)
    before = gather(table.tensors, pos)
    seed, eps = (12345, 2, 9), float(F32(1e-3))
    for e in (eps, -2 * eps, eps):
        jb.jb_perturb(table, seed, e)
    torch.cuda.synchronize()
    after = gather(table.tensors, pos)
    scale = np.abs(as_f64(before)) + 2 * eps * np.abs(oracle.gaussian_at(seed, idx))
    ulp = np.ldexp(1.0, np.frexp(scale)[1] - 8)
    assert np.all(np.abs(as_f64(after) - as_f64(before)) <= 1.5 * ulp)
    del table
    free_cuda()


def test_toy_spsa_run_matches_oracle(jb):
    """Toy quadratic, 2^20 fp32, K = 4 machines, 8 steps of Algorithm 1."""
    from oracle import spsa
    toy = synthetic.toy_quadratic(1 << 20)
    mids = synthetic.toy_machine_ids()
    eps, lr, qs, steps = float(F32(1e-3)), float(F32(1e-4)), 1.0, 8
    # the oracle's run, free from the same inputs
    theta_o, recs = spsa.spsa_run(toy.theta0, toy.a, toy.target, mids, steps, eps, lr, qs)
    # the same run on the GPU
    a = torch.from_numpy(toy.a).cuda()
    target = torch.from_numpy(toy.target).cuda()
    theta = to_device(toy.theta0)
    table = jb.ParamTable([theta], [0])
    loss = lambda: float((0.5 * a * (theta.double() - target) ** 2).sum())
    for t in range(steps):
        backup = theta.clone()
        seeds, codes, ghats = [], [], []
        for m in mids:
            s = (int(m), t, 0)
            theta.copy_(backup)
            jb.jb_perturb(table, s, eps)
            lp = loss()
            jb.jb_perturb(table, s, -2 * eps)
            lm = loss()
            g = (lp - lm) / (2 * eps)
            seeds.append(s)
            ghats.append(g)
            codes.append(jb.jb_quantize_grad(g, qs))
        theta.copy_(backup)
        jb.jb_apply_updates(table, seeds, codes, lr, float(len(seeds)), qs)
        r = recs[t]
        np.testing.assert_allclose(ghats, r.ghat, rtol=1e-3)
        assert codes == r.codes, (t, codes, r.codes)
    got = to_host(theta)
    # free-running: every step may add 2e-6 (|theta_t| + sum_k |c_k| max|z|), max|z| < 6
    csum = sum(abs(oracle.coefficient(c, lr, 4.0, qs)) for r in recs for c in r.codes)
    theta_max = np.maximum(np.abs(toy.theta0), np.abs(theta_o)).astype(np.float64) + 6 * csum
    d = np.abs(got.astype(np.float64) - theta_o.astype(np.float64))
    assert np.all(d <= 2e-6 * (steps * theta_max + 6 * csum))


def test_dynamic_membership_30b(jb):
    """OPT-30B-shaped bf16 (772 tensors, ~60 GB): 20 steps, 1..512 machines per step
    drawn from a pool of 1024 non-contiguous ids, denom = K_t; 2^22 sampled indices
    checked in two modes (Algorithm 1's gradient loop; Section 2, machines joining
    and leaving):
      stepwise      each step's oracle input is the GPU's theta at that step's start;
                    every sampled element is within one bf16 step of the oracle (R13:
                    beyond it only where the fp32 allowance of the operands admits it,
                    for at most BF16_WIDENED_SHARE of the elements of a step);
      free-running  the oracle runs all 20 steps from the same start; the bf16-step
                    histogram is printed and every element lies within the allowance
                    accumulated over the steps."""
    n_samples = 1 << 22
    table, pos, offs = _setup(jb, "opt-30b", "bf16", n_samples=n_samples)
    idx = global_index(offs, pos)
    before = gather(table.tensors, pos)
    start, free = before.copy(), before.copy()
    lr, qs = float(F32(1e-4)), 16.0
    Ks, wide = [], 0
    allowance = np.zeros(idx.size)
    for t, active in enumerate(synthetic.membership_schedule(20)):
        seeds = [(int(m), t, 0) for m in active]
        q = synthetic.byte_codes(len(seeds), 700 + t)
        K = len(seeds)
        Ks.append(K)
        jb.jb_apply_updates(table, seeds, q, lr, float(K), qs)
        after = gather(table.tensors, pos)
        # one oracle evaluation of sum c z and sum |c z| serves both modes
        delta, mag = oracle.update_delta_abs_at(idx, seeds, q, lr, float(K), qs)
        mark = len(WIDENED)
        check_theta(after, oracle.round_bf16(as_f64(before) + delta), np.abs(as_f64(before)) + mag,
                    f"30B stepwise t={t} K={K}")
        wide += WIDENED[mark][1]
        scale = np.abs(as_f64(free)) + mag
        allowance += np.ldexp(1.0, np.frexp(scale)[1] - 8) + 2e-6 * scale
        free = oracle.round_bf16(as_f64(free) + delta)
        before = after
    d = np.abs(bf16_ord(before) - bf16_ord(free))
    hist = np.bincount(np.minimum(d, 64).astype(np.int64))
    err = np.abs(as_f64(before) - as_f64(free))
    print(f"K_t = {Ks}; sampled {idx.size} of {sum(t.numel() for t in table.tensors)} "
          f"({idx.size / sum(t.numel() for t in table.tensors):.2e}); stepwise: {wide} element-steps "
          f"beyond one bf16 step of {idx.size * len(Ks)}; free-running bf16 step histogram "
          f"{hist.tolist()}; worst error / allowance {float((err / allowance).max()):.3f}")
    assert np.all(err <= allowance)
    assert not np.array_equal(before, start)
    del table
    free_cuda()
