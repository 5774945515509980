"""Host logic of bench.py that needs no GPU: the tensor groups of the end-to-end
pipeline (theta in pinned host memory, copied in and out group by group).

The split must be a partition of the tensors into exactly the requested number
of non-empty groups (fewer only when there are fewer tensors), and the groups at
both ends must be small, since their copies are the ones that compute cannot
hide."""
import importlib.util
import os

import numpy as np
import pytest

import synthetic

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def bench():
    spec = importlib.util.spec_from_file_location("bench", os.path.join(ROOT, "bench.py"))
    mod = importlib.util.module_from_spec(spec)
    spec.loader.exec_module(mod)
    return mod


class _Shape:
    def __init__(self, n):
        self.n = n

    def numel(self):
        return self.n


def _tensors(model):
    return [_Shape(int(np.prod(s.shape))) for s in synthetic.opt_tensors(model)]


@pytest.mark.parametrize("model", ["opt-125m", "opt-1.3b", "opt-13b", "opt-30b"])
@pytest.mark.parametrize("n_groups", [1, 2, 3, 5, 9, 16, 32, 64])
def test_e2e_split_is_a_partition(bench, model, n_groups):
    ts = _tensors(model)
    groups = bench.E2EPipeline.split(ts, n_groups)
    assert len(groups) == min(n_groups, len(ts))
    assert all(groups)
    assert sorted(i for g in groups for i in g) == list(range(len(ts)))


@pytest.mark.parametrize("model", ["opt-13b", "opt-30b"])
def test_e2e_split_ramps_at_both_ends(bench, model):
    ts = _tensors(model)
    total = sum(t.n for t in ts)
    groups = bench.E2EPipeline.split(ts, 16)
    share = [sum(ts[i].n for i in g) / total for g in groups]
    # a middle group holds about 1/12 of theta (16 groups, 4 ramp steps of
    # 1/16 .. 1/2 at each end); the end groups about 1/16 of that
    assert share[0] < 0.02 and share[-1] < 0.02, share
    assert max(share[4:-4]) < 0.15, share


def test_e2e_split_few_tensors(bench):
    ts = [_Shape(n) for n in (5, 1_000_000, 3)]
    for g in (1, 2, 3, 10):
        groups = bench.E2EPipeline.split(ts, g)
        assert len(groups) == min(g, 3) and all(groups)
        assert sorted(i for grp in groups for i in grp) == [0, 1, 2]
