"""The end-to-end pipeline of bench.py (theta in pinned host memory, tensor groups
copied in, stepped and copied out on three streams) leaves exactly the bits the
plain in-place calls on one device table give: any split of the table and any
overlap of copies with compute must change nothing."""
import importlib.util
import os

import numpy as np
import pytest

import synthetic

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def jb():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2306_10015_gb300 import build
    build.build()
    import paper_2306_10015_gb300 as pkg
    pkg.lib()
    return pkg


@pytest.fixture(scope="module")
def bench():
    spec = importlib.util.spec_from_file_location("bench", os.path.join(ROOT, "bench.py"))
    mod = importlib.util.module_from_spec(spec)
    spec.loader.exec_module(mod)
    return mod


@pytest.mark.parametrize("n_groups", [1, 5, 32])
def test_e2e_pipeline_matches_in_place_calls(jb, bench, n_groups):
    specs, tensors, offs = synthetic.opt_parameters("opt-125m", torch.bfloat16)
    ref = [t.clone() for t in tensors]
    stream = torch.cuda.current_stream()
    pipe = bench.E2EPipeline(jb, tensors, offs, stream, n_groups)
    del tensors
    K = 8
    mids = synthetic.machine_ids(K, 970)
    table = jb.ParamTable(ref, offs)
    for t in range(3):
        seeds = [(int(m), t, 0) for m in mids]
        q = synthetic.byte_codes(K, 970, t)
        s_own = (int(mids[0]), t, 0)
        pipe.step(s_own, seeds, q, 1e-3, 1e-4, 16.0)
        jb.jb_perturb(table, s_own, 1e-3, stream)
        jb.jb_perturb(table, s_own, -2e-3, stream)
        jb.jb_perturb(table, s_own, 1e-3, stream)
        jb.jb_apply_updates(table, seeds, q, 1e-4, 1.0, 16.0, stream)
    torch.cuda.synchronize()
    assert len(pipe.groups) == n_groups
    for h, r in zip(pipe.host_views, ref):
        assert torch.equal(h.view(torch.int16), r.cpu().view(torch.int16))
    # the parameters really moved
    moved = sum(int((h.view(torch.int16) != r0.cpu().view(torch.int16)).sum())
                for h, r0 in zip(pipe.host_views, synthetic.opt_parameters("opt-125m", torch.bfloat16)[1]))
    assert moved > 0
