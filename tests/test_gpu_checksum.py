"""The model checksum (ChecksumMatch, Algorithm 1): bit-exact against the oracle,
independent of the launch grid, and sensitive to any changed element."""
import numpy as np
import pytest

import oracle
import synthetic
from jbtest_util import to_device, to_host
from test_gpu_parity import LAYOUTS, download, make_layout, upload

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


def gpu_checksum(jb, table, grid=0):
    out = torch.zeros(1, dtype=torch.int64, device="cuda")
    jb.jb_checksum(table, out, grid_ctas=grid)
    torch.cuda.synchronize()
    return int(out.cpu().numpy().view(np.uint64)[0])


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
@pytest.mark.parametrize("kind", LAYOUTS)
def test_checksum_matches_oracle(jb, dtype, kind):
    vals, offs, shifts = make_layout(kind, dtype)
    table = upload(jb, vals, offs, shifts)
    assert gpu_checksum(jb, table) == oracle.checksum(vals, offs)


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_checksum_grid_independent_and_sensitive(jb, dtype):
    vals, offs, shifts = make_layout("ragged", dtype)
    table = upload(jb, vals, offs, shifts)
    ref = gpu_checksum(jb, table)
    for grid in (1, 7, 152, 1000):
        assert gpu_checksum(jb, table, grid) == ref
    t = table.tensors[5]
    raw = t.view(torch.int32 if dtype == "f32" else torch.int16)
    old = raw[17].clone()
    raw[17] ^= 1
    changed = gpu_checksum(jb, table)
    assert changed != ref
    host = download(table)
    assert changed == oracle.checksum(host, offs)
    raw[17] = old
    assert gpu_checksum(jb, table) == ref


def test_checksum_many_segments(jb):
    sizes = synthetic.ragged_sizes(1500, 300, 4)
    offs = synthetic.flat_offsets(sizes)
    vals = [oracle.round_bf16(synthetic.normal_values(n, 0.02, 5000 + i).astype(np.float64))
            for i, n in enumerate(sizes)]
    table = upload(jb, vals, offs, [0] * len(sizes))
    assert gpu_checksum(jb, table) == oracle.checksum(vals, offs)


def test_checksum_full_size_opt1p3b(jb):
    """The OPT-1.3B-shaped bf16 set (1.3e9 elements) against the oracle on its full copy."""
    specs, tensors, offs = synthetic.opt_parameters("opt-1.3b", torch.bfloat16)
    table = jb.ParamTable(tensors, offs)
    got = gpu_checksum(jb, table)
    host = [to_host(t) for t in tensors]
    assert got == oracle.checksum(host, offs)


def test_checksum_full_size_opt13b(jb):
    """The OPT-13B-shaped bf16 set (12.85e9 elements, the benchmark's launch). The
    checksum is a sum mod 2^64 of per-window terms, and a window never spans two
    tensors (flat offsets are multiples of 8 elements), so the whole-table value
    must equal the sum of the 644 one-tensor values; the token embedding, 8
    random tensors of >= 2^24 elements and random others (24 in all) are checked
    against the oracle on their full host copies."""
    specs, tensors, offs = synthetic.opt_parameters("opt-13b", torch.bfloat16)
    full = gpu_checksum(jb, jb.ParamTable(tensors, offs))
    per = [gpu_checksum(jb, jb.ParamTable([t], [fo])) for t, fo in zip(tensors, offs)]
    assert full == sum(per) % (1 << 64)
    rng = synthetic.rng(98)
    big = [i for i, t in enumerate(tensors) if t.numel() >= 1 << 24]
    picks = set(rng.choice(big, size=8, replace=False).tolist()) | {0}  # 0: the token embedding
    picks |= set(rng.choice(len(tensors), size=24 - len(picks), replace=False).tolist())
    for i in sorted(picks):
        assert per[i] == oracle.checksum([to_host(tensors[i])], [offs[i]]), int(i)
    print(f"checked against the oracle: {sum(tensors[i].numel() for i in picks)} elements "
          f"in {len(picks)} tensors")
    del tensors
    torch.cuda.empty_cache()
