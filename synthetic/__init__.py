"""Seeded synthetic inputs shared by the tests, the benchmark and the oracle checks.

This module holds no arithmetic of the method itself (no random-number stream
of the method, no Gaussian transform, no perturbation, no update, no byte
codec). It only builds workload shapes and draws input values with numpy's or
torch's own seeded generators, so that the CUDA path and the CPU oracle can be
fed identical bytes.

Workloads stand in for the paper's fine-tuning runs (OPT models on SST-2,
Section 3): the hot path depends only on the parameter count, the dtype, the
tensor sizes and the number of (seed, byte) pairs, so parameter sets are
shaped like OPT decoders and filled with synthetic values.
"""
from __future__ import annotations

import dataclasses
from typing import Iterator, List, Sequence, Tuple

import numpy as np

MASTER_SEED = 2306010015

# OPT decoder shapes: (layers, d_model, ffn, vocab, learned positions).
# OPT's learned position table has 2048 + 2 rows.
OPT_SHAPES = {
    "opt-125m": (12, 768, 3072, 50272, 2050),
    "opt-1.3b": (24, 2048, 8192, 50272, 2050),
    "opt-6.7b": (32, 4096, 16384, 50272, 2050),
    "opt-13b": (40, 5120, 20480, 50272, 2050),
    "opt-30b": (48, 7168, 28672, 50272, 2050),
}

# flat element index of tensor t starts at align_up(end of tensor t-1, FLAT_ALIGN)
FLAT_ALIGN = 8


@dataclasses.dataclass(frozen=True)
class TensorSpec:
    name: str
    shape: Tuple[int, ...]
    init: str  # "normal" (N(0, 0.02)), "ones" or "zeros"

    @property
    def numel(self) -> int:
        n = 1
        for s in self.shape:
            n *= s
        return n


def opt_tensors(model: str) -> List[TensorSpec]:
    """Parameter tensors of an OPT decoder in named_parameters() order.

    Per layer: q/k/v/out projections (weight + bias), attention LayerNorm,
    fc1, fc2 and the final LayerNorm of the block: 16 tensors. Plus token and
    position embeddings and the decoder's final LayerNorm; the LM head is
    tied to the token embedding. Total 16 L + 4 tensors.
    """
    L, d, F, V, P = OPT_SHAPES[model]
    out = [TensorSpec("embed_tokens.weight", (V, d), "normal"),
           TensorSpec("embed_positions.weight", (P, d), "normal")]
    for i in range(L):
        p = f"layers.{i}."
        for proj in ("k_proj", "v_proj", "q_proj", "out_proj"):
            out.append(TensorSpec(p + f"self_attn.{proj}.weight", (d, d), "normal"))
            out.append(TensorSpec(p + f"self_attn.{proj}.bias", (d,), "zeros"))
        out.append(TensorSpec(p + "self_attn_layer_norm.weight", (d,), "ones"))
        out.append(TensorSpec(p + "self_attn_layer_norm.bias", (d,), "zeros"))
        out.append(TensorSpec(p + "fc1.weight", (F, d), "normal"))
        out.append(TensorSpec(p + "fc1.bias", (F,), "zeros"))
        out.append(TensorSpec(p + "fc2.weight", (d, F), "normal"))
        out.append(TensorSpec(p + "fc2.bias", (d,), "zeros"))
        out.append(TensorSpec(p + "final_layer_norm.weight", (d,), "ones"))
        out.append(TensorSpec(p + "final_layer_norm.bias", (d,), "zeros"))
    out.append(TensorSpec("final_layer_norm.weight", (d,), "ones"))
    out.append(TensorSpec("final_layer_norm.bias", (d,), "zeros"))
    return out


def align_up(x: int, a: int) -> int:
    return (x + a - 1) // a * a


def flat_offsets(numels: Sequence[int], align: int = FLAT_ALIGN) -> List[int]:
    """Flat element index of the first element of each tensor."""
    offs, cur = [], 0
    for n in numels:
        offs.append(cur)
        cur = align_up(cur + n, align)
    return offs


def rng(*stream: int) -> np.random.Generator:
    """Independent numpy generator for one named input stream."""
    return np.random.default_rng(np.random.SeedSequence([MASTER_SEED, *stream]))


def machine_ids(n: int, *stream: int) -> np.ndarray:
    """n distinct random 64-bit machine identifiers (uint64)."""
    g = rng(101, *stream)
    ids = set()
    out = []
    while len(out) < n:
        v = int(g.integers(0, 2**64, dtype=np.uint64))
        if v not in ids:
            ids.add(v)
            out.append(v)
    return np.array(out, dtype=np.uint64)


def timestamp_ids(offsets_ns: Sequence[int], base_ns: int = 1_700_000_000_000_000_000) -> np.ndarray:
    """Machine start times in ns, used as machine identifiers (Section 2)."""
    return np.array([base_ns + o for o in offsets_ns], dtype=np.uint64)


def byte_codes(n: int, *stream: int) -> np.ndarray:
    """n one-byte projected-gradient codes uniform over all 256 values (int8)."""
    return rng(102, *stream).integers(-128, 128, size=n).astype(np.int8)


def normal_values(n: int, std: float, *stream: int, dtype=np.float32) -> np.ndarray:
    return (rng(103, *stream).standard_normal(n) * std).astype(dtype)


@dataclasses.dataclass
class ToyQuadratic:
    """Toy quadratic L(theta) = 0.5 * sum_i a_i (theta_i - theta*_i)^2."""
    theta0: np.ndarray   # float32, N(0, 1)
    a: np.ndarray        # float64, U(0.5, 2)
    target: np.ndarray   # float64, N(0, 1)


def toy_quadratic(n: int = 1 << 20) -> ToyQuadratic:
    g = rng(201)
    theta0 = g.standard_normal(n).astype(np.float32)
    a = g.uniform(0.5, 2.0, size=n)
    target = g.standard_normal(n)
    return ToyQuadratic(theta0, a, target)


def toy_machine_ids() -> np.ndarray:
    """Four machines whose start-time identifiers are not contiguous."""
    return timestamp_ids([0, 137, 9001, 31337])


def ragged_sizes(n_tensors: int, max_numel: int, *stream: int) -> List[int]:
    """Tensor sizes with odd lengths, including 1-element tensors."""
    g = rng(301, *stream)
    sizes = g.integers(1, max_numel + 1, size=n_tensors).tolist()
    if n_tensors > 2:
        sizes[0] = 1
        sizes[-1] = max(1, max_numel | 1)
    return [int(s) for s in sizes]


def membership_schedule(n_steps: int, pool: int = 1024, max_active: int = 512, *stream: int
                        ) -> Iterator[np.ndarray]:
    """Per-step active machine ids: count ~ U{1..max_active} from a fixed pool."""
    ids = machine_ids(pool, 401, *stream)
    g = rng(402, *stream)
    for _ in range(n_steps):
        m = int(g.integers(1, max_active + 1))
        yield np.sort(g.choice(ids, size=m, replace=False))


def opt_parameters(model: str, dtype, device="cuda", seed: int = MASTER_SEED):
    """OPT-shaped parameter tensors on `device`, one allocation per tensor.

    Weights and embeddings ~ N(0, 0.02), LayerNorm gains 1, biases 0, drawn
    with torch's own seeded generator on the device (input generation only).
    Returns (specs, tensors, flat_offsets).
    """
    import torch
    specs = opt_tensors(model)
    gen = torch.Generator(device=device)
    gen.manual_seed(seed)
    tensors = []
    for s in specs:
        t = torch.empty(s.numel, dtype=dtype, device=device)
        if s.init == "normal":
            t.normal_(0.0, 0.02, generator=gen)
        elif s.init == "ones":
            t.fill_(1.0)
        else:
            t.zero_()
        tensors.append(t)
    return specs, tensors, flat_offsets([s.numel for s in specs])


def sample_positions(numels: Sequence[int], n_samples: int, *stream: int) -> List[np.ndarray]:
    """Per-tensor sorted sample positions: the first and last element of every
    tensor plus n_samples positions drawn uniformly over all elements."""
    g = rng(501, *stream)
    total = int(sum(numels))
    flat = np.sort(g.integers(0, total, size=n_samples, dtype=np.int64))
    bounds = np.cumsum([0] + [int(n) for n in numels])
    out = []
    for i, n in enumerate(numels):
        lo, hi = np.searchsorted(flat, [bounds[i], bounds[i + 1]])
        p = np.concatenate([[0, int(n) - 1], flat[lo:hi] - bounds[i]])
        out.append(np.unique(p).astype(np.int64))
    return out
