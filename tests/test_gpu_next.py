"""The update read from the weight backup (restore fused, Algorithm 1) and the
multi-step replay of a late joiner (Appendix B): bitwise against the
composition of the basic calls they replace, and within tolerance against the
oracle."""
import numpy as np
import pytest

import oracle
import synthetic
from jbtest_util import as_f64, check_theta, to_host, update_scale
from test_gpu_parity import F32, LR, DENOM, QS, _pairs, download, make_layout, upload

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu


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


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
@pytest.mark.parametrize("kind", ["ragged", "phase"])
@pytest.mark.parametrize("K", [0, 1, 17])
@pytest.mark.parametrize("write_src", [False, True])
def test_apply_from_equals_copy_then_update(jb, dtype, kind, K, write_src):
    vals, offs, shifts = make_layout(kind, dtype)
    backup = upload(jb, vals, offs, shifts)
    theta = upload(jb, [np.zeros_like(v) for v in vals], offs, shifts[::-1])
    ref = upload(jb, vals, offs, shifts)
    seeds, q = _pairs(K, stream=3) if K else ([], np.zeros(0, np.int8))
    jb.jb_apply_updates_from(backup, theta, seeds, q, LR, DENOM, QS, write_src=write_src)
    jb.jb_apply_updates(ref, seeds, q, LR, DENOM, QS)
    sync()
    for v, b, t, r in zip(vals, download(backup), download(theta), download(ref)):
        assert np.array_equal(t, r)
        assert np.array_equal(b, r if write_src else v)


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_apply_from_in_place_and_oracle(jb, dtype):
    vals, offs, shifts = make_layout("ragged", dtype)
    a = upload(jb, vals, offs, shifts)
    b = upload(jb, vals, offs, shifts)
    seeds, q = _pairs(9, stream=4)
    jb.jb_apply_updates_from(a, a, seeds, q, LR, DENOM, QS)
    jb.jb_apply_updates(b, seeds, q, LR, DENOM, QS)
    sync()
    for v, fo, x, y in zip(vals, offs, download(a), download(b)):
        assert np.array_equal(x, y)
        idx = np.arange(fo, fo + v.size, dtype=np.uint64)
        check_theta(x, oracle.update(v, fo, seeds, q, LR, DENOM, QS),
                    update_scale(v, idx, seeds, q, LR, DENOM, QS), "apply_from")


def _steps(sizes, stream):
    steps = []
    for t, K in enumerate(sizes):
        mids = synthetic.machine_ids(max(K, 1), 800 + stream, t)[:K]
        seeds = [(int(m), t, int(j % 2)) for j, m in enumerate(mids)]
        q = synthetic.byte_codes(K, 800 + stream, t)
        lr = float(F32(1e-3 / (1 + t)))
        denom = float(F32(max(K, 1)))
        steps.append((seeds, q, lr, denom))
    return steps


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
@pytest.mark.parametrize("kind", ["ragged", "phase", "high"])
def test_replay_equals_sequential_calls(jb, dtype, kind):
    vals, offs, shifts = make_layout(kind, dtype)
    a = upload(jb, vals, offs, shifts)
    b = upload(jb, vals, offs, shifts)
    steps = _steps([3, 0, 17, 1, 40, 5], 1)
    jb.jb_replay_updates(a, steps, QS)
    for seeds, q, lr, denom in steps:
        jb.jb_apply_updates(b, seeds, q, lr, denom, QS)
    sync()
    for x, y in zip(download(a), download(b)):
        assert np.array_equal(x, y)


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_replay_across_launches(jb, dtype):
    """1200 pairs in 40 steps: three launches of at most 512 pairs."""
    vals, offs, shifts = make_layout("ragged", dtype)
    vals, offs, shifts = vals[:8], offs[:8], shifts[:8]
    a = upload(jb, vals, offs, shifts)
    b = upload(jb, vals, offs, shifts)
    steps = _steps([30] * 40, 2)
    jb.jb_replay_updates(a, steps, QS)
    for seeds, q, lr, denom in steps:
        jb.jb_apply_updates(b, seeds, q, lr, denom, QS)
    sync()
    for x, y in zip(download(a), download(b)):
        assert np.array_equal(x, y)


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_replay_against_oracle(jb, dtype):
    vals, offs, shifts = make_layout("phase", dtype)
    a = upload(jb, vals, offs, shifts)
    steps = _steps([4, 9, 2], 3)
    jb.jb_replay_updates(a, steps, QS)
    sync()
    for v, fo, got in zip(vals, offs, download(a)):
        idx = np.arange(fo, fo + v.size, dtype=np.uint64)
        want, allow = v, np.zeros(v.size)
        for seeds, q, lr, denom in steps:
            scale = update_scale(want, idx, seeds, q, lr, denom, QS)
            if dtype == "bf16":
                allow += np.ldexp(1.0, np.frexp(scale)[1] - 8) + 2e-6 * scale
            else:
                allow += 2e-6 * scale
            want = oracle.update(want, fo, seeds, q, lr, denom, QS)
        err = np.abs(as_f64(got) - as_f64(want))
        assert np.all(err <= allow + 2.0**-133), float((err / (allow + 1e-300)).max())
