"""C-ABI checks that need no GPU: exported symbols, the host byte codec against
the oracle (bit-exact), and argument validation, which happens before anything
touches CUDA. Fake device addresses are never dereferenced: every call here
returns an error (or a no-op) before a launch."""
import ctypes
import math
import os
import re
import subprocess

import numpy as np
import pytest

import oracle
import synthetic

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def jb():
    from paper_2306_10015_gb300 import build
    build.build()
    import paper_2306_10015_gb300 as pkg
    pkg.lib()
    return pkg


def declared_functions():
    with open(os.path.join(ROOT, "include", "jb.h")) as f:
        text = f.read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(jb_[a-z_0-9]+)\s*\(", text)))


def test_library_exports_every_declared_symbol(jb):
    names = declared_functions()
    assert "jb_perturb" in names and "jb_apply_updates" in names
    assert "jb_quantize_grad" in names and "jb_dequantize_grad" in names
    out = subprocess.run(["nm", "-D", "--defined-only", jb.build.LIB], capture_output=True,
                         text=True, check=True).stdout
    exported = {ln.split()[-1] for ln in out.splitlines() if ln.strip()}
    missing = [n for n in names if n not in exported]
    assert not missing, missing
    for n in names:
        assert hasattr(jb.lib(), n)


def test_status_strings(jb):
    for rc in range(-8, 1):
        assert jb.jb_status_string(rc) not in ("", "unknown status")
    assert jb.jb_status_string(17) == "unknown status"


@pytest.mark.parametrize("S", [1.0, 8.0, 16.0, float(np.float32(3.7))])
def test_quantize_bit_exact_vs_oracle(jb, S):
    g = np.concatenate([np.logspace(-8, 70, 4000), -np.logspace(-8, 70, 4000),
                        [0.0, -0.0, 1e-300, 5e-324]])
    # values on and around every rounding boundary expm1((n + 1/2) / S)
    b = np.expm1((np.arange(127) + 0.5) / S)
    g = np.concatenate([g, b, np.nextafter(b, 0), np.nextafter(b, np.inf), -b])
    for v in g:
        assert jb.jb_quantize_grad(float(v), S) == oracle.quantize(float(v), S), v
    for v in (float("nan"), float("inf"), -float("inf")):
        assert jb.jb_quantize_grad(v, S) == oracle.quantize(v, S)


@pytest.mark.parametrize("S", [1.0, 8.0, 16.0, float(np.float32(0.37))])
def test_dequantize_bit_exact_vs_oracle(jb, S):
    for q in range(-128, 128):
        with np.errstate(over="ignore"):
            want = np.float32(oracle.dequantize(q, S))
        got = np.float32(jb.jb_dequantize_grad(q, S))
        assert got.tobytes() == want.tobytes(), q


def test_codec_rejects_bad_scale(jb):
    for S in (0.0, -1.0, float("nan"), float("inf")):
        with pytest.raises(jb.JbError):
            jb.jb_quantize_grad(1.0, S)
        with pytest.raises(jb.JbError):
            jb.jb_dequantize_grad(3, S)


# --- argument validation (returns before any CUDA call) -------------------------

def _segs(jb, spec):
    arr = (jb.jb_segment * len(spec))()
    for i, (p, n, fo) in enumerate(spec):
        arr[i] = jb.jb_segment(p, n, fo)
    return arr


def _perturb(jb, segs, n, dtype=0, eps=1e-3):
    return jb.lib().jb_perturb(segs, n, dtype, jb.jb_seed(1, 0, 0), eps, None)


def _update(jb, segs, n, seeds, q, dtype=0, lr=1e-3, denom=1.0, qscale=16.0, K=None):
    s = jb.seeds_array(seeds)
    qa = np.asarray(q, dtype=np.int8)
    K = len(s) if K is None else K
    return jb.lib().jb_apply_updates(segs, n, dtype, ctypes.c_void_p(s.ctypes.data if len(s) else None),
                                     ctypes.c_void_p(qa.ctypes.data if len(qa) else None), K, lr,
                                     denom, qscale, None)


FAKE = 0x7F0000000000  # never dereferenced


def test_empty_calls_are_noops(jb):
    assert _perturb(jb, None, 0) == 0
    assert _perturb(jb, _segs(jb, [(0, 0, 0)]), 1) == 0           # empty segment, NULL ptr
    assert _update(jb, _segs(jb, [(FAKE, 100, 0)]), 1, [], []) == 0  # K = 0


def test_invalid_arguments(jb):
    E = {"inv": -1, "dtype": -2, "mis": -3, "dup": -4, "range": -6, "many": -7}
    ok = _segs(jb, [(FAKE, 100, 0)])
    assert _perturb(jb, ok, 1, dtype=2) == E["dtype"]
    assert _perturb(jb, ok, -1) == E["inv"]
    assert _perturb(jb, None, 3) == E["inv"]
    assert _perturb(jb, _segs(jb, [(0, 5, 0)]), 1) == E["inv"]                 # NULL, numel > 0
    assert _perturb(jb, _segs(jb, [(FAKE + 2, 5, 0)]), 1, dtype=0) == E["mis"]  # fp32 needs 4 B
    assert _perturb(jb, _segs(jb, [(FAKE + 1, 5, 0)]), 1, dtype=1) == E["mis"]  # bf16 needs 2 B
    assert _perturb(jb, ok, 1, eps=float("nan")) == E["inv"]
    # overlap in global index, overlap in memory
    assert _perturb(jb, _segs(jb, [(FAKE, 10, 0), (FAKE + 4096, 10, 9)]), 2) == E["inv"]
    assert _perturb(jb, _segs(jb, [(FAKE, 10, 0), (FAKE + 36, 10, 100)]), 2) == E["inv"]
    assert _perturb(jb, _segs(jb, [(FAKE, 10, (1 << 62) - 5)]), 1) == E["inv"]
    # a segment that would run past the end of the address space, including the
    # case where numel * sizeof(T) itself is 2^64
    assert _perturb(jb, _segs(jb, [(16, 1 << 62, 0)]), 1, dtype=0) == E["inv"]
    assert _perturb(jb, _segs(jb, [((1 << 64) - 64, 100, 0)]), 1, dtype=1) == E["inv"]
    seeds = [(1, 0, 0), (2, 0, 0)]
    assert _update(jb, ok, 1, seeds + [(1, 0, 0)], [1, 2, 3]) == E["dup"]
    assert _update(jb, ok, 1, seeds, [1, 2], K=-1) == E["inv"]
    assert _update(jb, ok, 1, seeds, [1, 2], denom=0.0) == E["inv"]
    assert _update(jb, ok, 1, seeds, [1, 2], qscale=0.0) == E["inv"]
    assert _update(jb, ok, 1, seeds, [1, 2], lr=float("inf")) == E["inv"]
    # expm1(127) overflows fp32: coefficient not representable
    assert _update(jb, ok, 1, seeds, [127, 2], lr=1.0, qscale=1.0) == E["range"]
    K = jb.jb_max_seeds_per_call() + 1
    many = [(i + 1, 0, 0) for i in range(K)]
    assert _update(jb, ok, 1, many, [1] * K) == E["many"]


def test_python_table_rejects_cpu_tensors(jb):
    import torch
    with pytest.raises(ValueError):
        jb.ParamTable([torch.zeros(4)])
    with pytest.raises(TypeError):
        jb.ParamTable([torch.zeros(4, dtype=torch.float16)])


def test_default_flat_offsets(jb):
    assert jb.default_flat_offsets([5, 8, 1, 9]) == [0, 8, 16, 24]
    assert jb.default_flat_offsets([5, 8, 1, 9]) == synthetic.flat_offsets([5, 8, 1, 9])


def test_opt_shapes_match_known_parameter_counts():
    counts = {"opt-125m": 125_239_296, "opt-1.3b": 1_315_758_080, "opt-13b": 12_853_473_280,
              "opt-30b": 29_974_540_288}
    for name, n in counts.items():
        t = synthetic.opt_tensors(name)
        L = synthetic.OPT_SHAPES[name][0]
        assert sum(x.numel for x in t) == n
        assert len(t) == 16 * L + 4


def test_apply_from_and_replay_validation(jb):
    import ctypes as C
    E = {"inv": -1, "dup": -4, "many": -7}
    src = _segs(jb, [(FAKE, 100, 0), (FAKE + 4096, 50, 104)])
    s = jb.seeds_array([(1, 0, 0), (2, 0, 0)])
    q = np.array([3, 4], dtype=np.int8)
    sp, qp = C.c_void_p(s.ctypes.data), C.c_void_p(q.ctypes.data)
    L = jb.lib()
    call = lambda dst, K=2: L.jb_apply_updates_from(src, dst, 2, 0, sp, qp, K, 1e-3, 1.0, 16.0, 0, None)
    assert call(None) == E["inv"]
    assert call(_segs(jb, [(FAKE + 8192, 100, 0), (FAKE + 16384, 49, 104)])) == E["inv"]  # numel
    assert call(_segs(jb, [(FAKE + 8192, 100, 1), (FAKE + 16384, 50, 104)])) == E["inv"]  # offset
    assert call(_segs(jb, [(FAKE + 200, 100, 0), (FAKE + 16384, 50, 104)])) == E["inv"]   # overlaps src
    assert call(_segs(jb, [(FAKE + 8192, 100, 0), (FAKE + 8200, 50, 104)])) == E["inv"]   # dsts overlap
    assert call(_segs(jb, [(FAKE + 8192, 100, 0), (FAKE + 16384, 50, 104)]), K=-1) == E["inv"]
    dup = jb.seeds_array([(1, 0, 0), (1, 0, 0)])
    assert L.jb_apply_updates_from(src, src, 2, 0, C.c_void_p(dup.ctypes.data), qp, 2, 1e-3, 1.0,
                                   16.0, 0, None) == E["dup"]
    sizes = np.array([1, 1], dtype=np.int32)
    lr = np.array([1e-3, 1e-3], dtype=np.float32)
    den = np.array([1.0, 0.0], dtype=np.float32)
    replay = lambda sz, d: L.jb_replay_updates(src, 2, 0, sp, qp, C.c_void_p(sz.ctypes.data), len(sz),
                                               C.c_void_p(lr.ctypes.data), C.c_void_p(d.ctypes.data),
                                               16.0, None)
    assert replay(sizes, den) == E["inv"]                                  # denom 0 in step 1
    assert replay(np.array([1, -1], np.int32), np.ones(2, np.float32)) == E["inv"]
    big = np.array([600, 0], np.int32)
    assert replay(big, np.ones(2, np.float32)) == E["many"]                # one step > 512 pairs
    # two equal seeds in different steps are legal (only a step must be duplicate-free):
    # validation passes and the call reaches the launch, which has no device here


def test_checksum_validation(jb):
    import ctypes as C
    src = _segs(jb, [(FAKE, 100, 0)])
    L = jb.lib()
    assert L.jb_checksum(src, 1, 0, None, None) == -1
    assert L.jb_checksum(src, 1, 0, C.c_void_p(FAKE + 4), None) == -3
    assert L.jb_checksum(src, 1, 3, C.c_void_p(FAKE), None) == -2


def test_q4_levels_match_oracle_and_validation(jb):
    import ctypes as C
    assert np.array_equal(jb.jb_q4_levels(), oracle.q4_levels())
    L = jb.lib()
    seg = (jb.jb_q4_segment * 1)()
    seg[0] = jb.jb_q4_segment(FAKE, FAKE + 4096, 100, 8)
    assert L.jb_perturb_q4(seg, 1, jb.jb_seed(1, 0, 0), float("nan"), None) == -1
    seg[0] = jb.jb_q4_segment(FAKE + 4, FAKE + 4096, 100, 8)       # codes not 8-byte aligned
    assert L.jb_perturb_q4(seg, 1, jb.jb_seed(1, 0, 0), 1e-3, None) == -3
    seg[0] = jb.jb_q4_segment(FAKE, FAKE + 4096, 100, 6)           # flat offset not a multiple of 4
    assert L.jb_perturb_q4(seg, 1, jb.jb_seed(1, 0, 0), 1e-3, None) == -3
    seg[0] = jb.jb_q4_segment(FAKE, FAKE + 40, 100, 8)             # scales overlap the codes
    assert L.jb_perturb_q4(seg, 1, jb.jb_seed(1, 0, 0), 1e-3, None) == -1
    seg[0] = jb.jb_q4_segment(0, FAKE, 100, 8)
    assert L.jb_perturb_q4(seg, 1, jb.jb_seed(1, 0, 0), 1e-3, None) == -1
    seg[0] = jb.jb_q4_segment(FAKE, FAKE + 4098, 100, 8)           # scale not 4-byte aligned
    assert L.jb_perturb_q4(seg, 1, jb.jb_seed(1, 0, 0), 1e-3, None) == -3
    seg[0] = jb.jb_q4_segment(FAKE, FAKE + 4096, 100, (1 << 62) - 96)  # index range past 2^62
    assert L.jb_perturb_q4(seg, 1, jb.jb_seed(1, 0, 0), 1e-3, None) == -1
    assert L.jb_perturb_q4(seg, -1, jb.jb_seed(1, 0, 0), 1e-3, None) == -1
    two = (jb.jb_q4_segment * 2)()
    two[0] = jb.jb_q4_segment(FAKE, FAKE + 4096, 100, 8)
    two[1] = jb.jb_q4_segment(FAKE + 8192, FAKE + 12288, 100, 104)  # index ranges overlap
    assert L.jb_perturb_q4(two, 2, jb.jb_seed(1, 0, 0), 1e-3, None) == -1
    two[0] = jb.jb_q4_segment(FAKE + 4, FAKE + 2, 0, 6)             # empty tensors are skipped,
    two[1] = jb.jb_q4_segment(0, 0, 0, 0)                           # unchecked: nothing to launch
    assert L.jb_perturb_q4(two, 2, jb.jb_seed(1, 0, 0), 1e-3, None) == 0


def test_debug_hooks_check_alignment(jb):
    """The test hooks refuse buffers their kernels could not store to or load from."""
    L, seed = jb.lib(), jb.jb_seed(1, 2, 3)
    assert L.jb_debug_philox(seed, 0, 4, ctypes.c_void_p(FAKE + 8), None) == -3
    assert L.jb_debug_gaussian(seed, 0, 4, ctypes.c_void_p(FAKE + 2), None) == -3
    assert L.jb_debug_box_muller(ctypes.c_void_p(FAKE + 1), 4, ctypes.c_void_p(FAKE), None) == -3
    assert L.jb_debug_box_muller(ctypes.c_void_p(FAKE), 4, ctypes.c_void_p(FAKE + 2), None) == -3
    assert L.jb_debug_gaussian(seed, 0, (1 << 38) + 1, ctypes.c_void_p(FAKE), None) == -1
    assert L.jb_debug_gaussian(seed, 0, 4, None, None) == -1


def test_philox_fold_validation(jb):
    """The generator-only hook refuses a missing, misaligned or oversized request
    before anything is enqueued."""
    L, seed = jb.lib(), jb.jb_seed(1, 2, 3)
    assert L.jb_debug_philox_fold(seed, 0, 4, None, None) == -1
    assert L.jb_debug_philox_fold(seed, 0, 4, ctypes.c_void_p(FAKE + 2), None) == -3
    assert L.jb_debug_philox_fold(seed, 0, (1 << 46) + 1, ctypes.c_void_p(FAKE), None) == -1
    assert L.jb_debug_philox_fold(seed, (1 << 60) + 1, 4, ctypes.c_void_p(FAKE), None) == -1
