"""Python binding of libjb, the sm_103a seeded-perturbation library.

Argument marshalling only: every element-wise step runs in the CUDA kernels
behind the C ABI of ``include/jb.h``; PyTorch supplies device memory and
streams. The functions keep the C names:

* ``jb_perturb``        PerturbParameters(theta, eps, s) (Algorithm 1, subroutine)
* ``jb_apply_updates``  the fused K-pair step update (Section 2; Algorithm 1)
* ``jb_apply_updates_from``  the same update read from the weight backup, with the
  restore of Algorithm 1 fused in
* ``jb_replay_updates``  several steps' updates in one pass (a late joiner's
  catch-up, Appendix B)
* ``jb_checksum``  the model hash of ChecksumMatch (Algorithm 1)
* ``jb_perturb_q4``  the perturbation of 4-bit weights (Section 3)
* ``jb_quantize_grad`` / ``jb_dequantize_grad``  the one-byte projected
  gradient (Section 3, Training Speed)

There is no CPU fallback: if ``libjb.so`` is missing, loading it raises.
"""
from __future__ import annotations

import ctypes
import os
import threading
from typing import Iterable, List, Optional, Sequence

import numpy as np

from .build import LIB as _LIB_PATH

JB_OK = 0
JB_F32, JB_BF16 = 0, 1

# Memory layout of jb_seed (16 bytes); arrays of it are passed without copying.
SEED_DTYPE = np.dtype([("machine_id", "<u8"), ("step", "<u4"), ("sample_id", "<u4")])

FLAT_ALIGN = 8


class JbError(RuntimeError):
    def __init__(self, status: int, message: str):
        super().__init__(f"libjb status {status}: {message}")
        self.status = status


class jb_segment(ctypes.Structure):
    _fields_ = [("ptr", ctypes.c_void_p), ("numel", ctypes.c_uint64),
                ("flat_offset", ctypes.c_uint64)]


class jb_q4_segment(ctypes.Structure):
    _fields_ = [("codes", ctypes.c_void_p), ("scale", ctypes.c_void_p), ("numel", ctypes.c_uint64),
                ("flat_offset", ctypes.c_uint64)]


class jb_seed(ctypes.Structure):
    _fields_ = [("machine_id", ctypes.c_uint64), ("step", ctypes.c_uint32),
                ("sample_id", ctypes.c_uint32)]


_lock = threading.Lock()
_lib: Optional[ctypes.CDLL] = None


def lib() -> ctypes.CDLL:
    """The loaded libjb.so. Raises if it has not been built."""
    global _lib
    with _lock:
        if _lib is None:
            if not os.path.exists(_LIB_PATH):
                raise RuntimeError(
                    f"libjb.so not found at {_LIB_PATH}; build it with "
                    "`python -m paper_2306_10015_gb300.build` (needs nvcc)")
            L = ctypes.CDLL(_LIB_PATH)
            vp, i32, u64, f32 = ctypes.c_void_p, ctypes.c_int, ctypes.c_uint64, ctypes.c_float
            L.jb_perturb.argtypes = [vp, i32, i32, jb_seed, f32, vp]
            L.jb_perturb_with_grid.argtypes = [vp, i32, i32, jb_seed, f32, i32, vp]
            L.jb_apply_updates.argtypes = [vp, i32, i32, vp, vp, i32, f32, f32, f32, vp]
            L.jb_apply_updates_with_grid.argtypes = [vp, i32, i32, vp, vp, i32, f32, f32, f32,
                                                     i32, vp]
            L.jb_apply_updates_from.argtypes = [vp, vp, i32, i32, vp, vp, i32, f32, f32, f32,
                                                i32, vp]
            L.jb_replay_updates.argtypes = [vp, i32, i32, vp, vp, vp, i32, vp, vp, f32, vp]
            L.jb_perturb_q4.argtypes = [vp, i32, jb_seed, f32, vp]
            L.jb_q4_levels.argtypes = [vp]
            L.jb_checksum.argtypes = [vp, i32, i32, vp, vp]
            L.jb_checksum_with_grid.argtypes = [vp, i32, i32, vp, i32, vp]
            L.jb_quantize_grad.argtypes = [ctypes.c_double, f32, ctypes.POINTER(ctypes.c_int8)]
            L.jb_dequantize_grad.argtypes = [ctypes.c_int8, f32, ctypes.POINTER(ctypes.c_float)]
            L.jb_max_seeds_per_call.argtypes = []
            L.jb_status_string.argtypes = [i32]
            L.jb_status_string.restype = ctypes.c_char_p
            L.jb_debug_philox.argtypes = [jb_seed, u64, u64, vp, vp]
            L.jb_debug_philox_fold.argtypes = [jb_seed, u64, u64, vp, vp]
            L.jb_debug_gaussian.argtypes = [jb_seed, u64, u64, vp, vp]
            L.jb_debug_box_muller.argtypes = [vp, u64, vp, vp]
            for f in ("jb_perturb", "jb_perturb_with_grid", "jb_apply_updates",
                      "jb_apply_updates_with_grid", "jb_apply_updates_from", "jb_replay_updates",
                      "jb_checksum", "jb_checksum_with_grid", "jb_perturb_q4", "jb_q4_levels",
                      "jb_quantize_grad", "jb_dequantize_grad",
                      "jb_max_seeds_per_call", "jb_debug_philox", "jb_debug_philox_fold",
                      "jb_debug_gaussian",
                      "jb_debug_box_muller"):
                getattr(L, f).restype = i32
            _lib = L
    return _lib


def jb_status_string(status: int) -> str:
    return lib().jb_status_string(int(status)).decode()


def _check(rc: int) -> None:
    if rc != JB_OK:
        raise JbError(rc, jb_status_string(rc))


def _stream(stream) -> ctypes.c_void_p:
    if stream is None:
        import torch
        return ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)
    if isinstance(stream, int):
        return ctypes.c_void_p(stream)
    return ctypes.c_void_p(stream.cuda_stream)


def _seed(s) -> jb_seed:
    if isinstance(s, jb_seed):
        return s
    if isinstance(s, np.void):
        return jb_seed(int(s["machine_id"]), int(s["step"]), int(s["sample_id"]))
    m, t, j = s
    return jb_seed(int(m), int(t), int(j))


def seeds_array(seeds) -> np.ndarray:
    """Seeds as a contiguous jb_seed array (machine_id, step, sample_id)."""
    if isinstance(seeds, np.ndarray) and seeds.dtype == SEED_DTYPE:
        return np.ascontiguousarray(seeds)
    out = np.zeros(len(seeds), dtype=SEED_DTYPE)
    for i, s in enumerate(seeds):
        out[i] = (int(s[0]), int(s[1]), int(s[2]))
    return out


def default_flat_offsets(numels: Sequence[int], align: int = FLAT_ALIGN) -> List[int]:
    """flat_offset of tensor t = align_up(flat_offset of t-1 + numel of t-1, align)."""
    offs, cur = [], 0
    for n in numels:
        offs.append(cur)
        cur = (cur + int(n) + align - 1) // align * align
    return offs


class ParamTable:
    """Segment table (jb_segment array) over CUDA tensors of one dtype.

    Holds references to the tensors so their memory stays alive. Element i of
    tensor t has global index flat_offsets[t] + i; every replica must build the
    table with the same offsets.
    """

    def __init__(self, tensors: Iterable, flat_offsets: Optional[Sequence[int]] = None):
        import torch
        self.tensors = list(tensors)
        if not self.tensors:
            raise ValueError("empty parameter list")
        dt = self.tensors[0].dtype
        if dt == torch.float32:
            self.dtype = JB_F32
        elif dt == torch.bfloat16:
            self.dtype = JB_BF16
        else:
            raise TypeError(f"parameters must be float32 or bfloat16, got {dt}")
        for t in self.tensors:
            if t.dtype != dt or not t.is_cuda or not t.is_contiguous():
                raise ValueError("parameters must be contiguous CUDA tensors of one dtype")
        numels = [t.numel() for t in self.tensors]
        self.flat_offsets = (list(flat_offsets) if flat_offsets is not None
                             else default_flat_offsets(numels))
        if len(self.flat_offsets) != len(self.tensors):
            raise ValueError("one flat offset per tensor")
        n = len(self.tensors)
        self.segments = (jb_segment * n)()
        for i, (t, fo) in enumerate(zip(self.tensors, self.flat_offsets)):
            self.segments[i] = jb_segment(t.data_ptr(), t.numel(), int(fo))
        self.numel = sum(numels)
        self.n_segments = n

    @classmethod
    def from_module(cls, module, flat_offsets=None) -> "ParamTable":
        return cls([p.data for _, p in module.named_parameters()], flat_offsets)


def jb_perturb(table: ParamTable, seed, eps: float, stream=None, grid_ctas: int = 0) -> None:
    """theta <- theta + eps z(seed), in place on `stream` (asynchronous)."""
    L = lib()
    if grid_ctas:
        rc = L.jb_perturb_with_grid(table.segments, table.n_segments, table.dtype, _seed(seed),
                                    float(eps), int(grid_ctas), _stream(stream))
    else:
        rc = L.jb_perturb(table.segments, table.n_segments, table.dtype, _seed(seed), float(eps),
                          _stream(stream))
    _check(rc)


def jb_apply_updates(table: ParamTable, seeds, q, lr: float, denom: float, qscale: float,
                     stream=None, grid_ctas: int = 0) -> None:
    """theta <- theta - (lr / denom) sum_k deq(q_k) z(seed_k), one pass, in place."""
    s = seeds_array(seeds)
    qa = np.ascontiguousarray(np.asarray(q, dtype=np.int8))
    if qa.shape[0] != s.shape[0]:
        raise ValueError("one byte code per seed")
    K = s.shape[0]
    sp = ctypes.c_void_p(s.ctypes.data if K else None)
    qp = ctypes.c_void_p(qa.ctypes.data if K else None)
    L = lib()
    if grid_ctas:
        rc = L.jb_apply_updates_with_grid(table.segments, table.n_segments, table.dtype, sp, qp, K,
                                          float(lr), float(denom), float(qscale), int(grid_ctas),
                                          _stream(stream))
    else:
        rc = L.jb_apply_updates(table.segments, table.n_segments, table.dtype, sp, qp, K,
                                float(lr), float(denom), float(qscale), _stream(stream))
    _check(rc)


def jb_apply_updates_from(src: ParamTable, dst: ParamTable, seeds, q, lr: float, denom: float,
                          qscale: float, write_src: bool = False, stream=None) -> None:
    """dst <- src - (lr / denom) sum_k deq(q_k) z(seed_k) in one pass (restore fused)."""
    if src.n_segments != dst.n_segments or src.dtype != dst.dtype:
        raise ValueError("source and destination tables differ")
    s = seeds_array(seeds)
    qa = np.ascontiguousarray(np.asarray(q, dtype=np.int8))
    if qa.shape[0] != s.shape[0]:
        raise ValueError("one byte code per seed")
    K = s.shape[0]
    _check(lib().jb_apply_updates_from(
        src.segments, dst.segments, src.n_segments, src.dtype,
        ctypes.c_void_p(s.ctypes.data if K else None), ctypes.c_void_p(qa.ctypes.data if K else None),
        K, float(lr), float(denom), float(qscale), int(bool(write_src)), _stream(stream)))


def jb_replay_updates(table: ParamTable, steps, qscale: float, stream=None) -> None:
    """Apply several steps' updates in order, in place; steps = [(seeds, q, lr, denom), ...]."""
    seeds = [seeds_array(st[0]) for st in steps]
    codes = [np.asarray(st[1], dtype=np.int8) for st in steps]
    sizes = np.array([len(x) for x in seeds], dtype=np.int32)
    if any(len(c) != n for c, n in zip(codes, sizes)):
        raise ValueError("one byte code per seed")
    s = np.ascontiguousarray(np.concatenate(seeds) if len(seeds) else np.zeros(0, SEED_DTYPE))
    qa = np.ascontiguousarray(np.concatenate(codes) if len(codes) else np.zeros(0, np.int8))
    lr = np.array([float(st[2]) for st in steps], dtype=np.float32)
    denom = np.array([float(st[3]) for st in steps], dtype=np.float32)
    T = len(steps)
    ptr = lambda a: ctypes.c_void_p(a.ctypes.data if a.size else None)
    _check(lib().jb_replay_updates(table.segments, table.n_segments, table.dtype, ptr(s), ptr(qa),
                                   ptr(sizes), T, ptr(lr), ptr(denom), float(qscale),
                                   _stream(stream)))


class Q4Table:
    """jb_q4_segment array over 4-bit tensors: (codes uint8 CUDA tensor, scales float32 CUDA
    tensor, numel) triples; flat offsets default to the jb_segment rule."""

    def __init__(self, tensors, flat_offsets: Optional[Sequence[int]] = None):
        self.tensors = list(tensors)
        numels = [int(n) for _, _, n in self.tensors]
        self.flat_offsets = (list(flat_offsets) if flat_offsets is not None
                             else default_flat_offsets(numels))
        n = len(self.tensors)
        self.segments = (jb_q4_segment * n)()
        for i, ((codes, scale, numel), fo) in enumerate(zip(self.tensors, self.flat_offsets)):
            if codes.numel() < (numel + 1) // 2 or scale.numel() < (numel + 63) // 64:
                raise ValueError("codes or scales too short for numel")
            self.segments[i] = jb_q4_segment(codes.data_ptr(), scale.data_ptr(), int(numel), int(fo))
        self.n_segments = n


def jb_perturb_q4(table: "Q4Table", seed, eps: float, stream=None) -> None:
    """4-bit weights: dequantize, add eps z(seed), quantize again, in place."""
    _check(lib().jb_perturb_q4(table.segments, table.n_segments, _seed(seed), float(eps),
                               _stream(stream)))


def jb_q4_levels() -> np.ndarray:
    out = np.empty(16, dtype=np.float32)
    _check(lib().jb_q4_levels(out.ctypes.data))
    return out


def jb_checksum(table: ParamTable, out, stream=None, grid_ctas: int = 0) -> None:
    """out (CUDA int64 tensor, one element) <- the model checksum, on `stream`."""
    L = lib()
    if grid_ctas:
        rc = L.jb_checksum_with_grid(table.segments, table.n_segments, table.dtype, out.data_ptr(),
                                     int(grid_ctas), _stream(stream))
    else:
        rc = L.jb_checksum(table.segments, table.n_segments, table.dtype, out.data_ptr(),
                           _stream(stream))
    _check(rc)


def jb_quantize_grad(g: float, qscale: float = 1.0) -> int:
    out = ctypes.c_int8()
    _check(lib().jb_quantize_grad(float(g), float(qscale), ctypes.byref(out)))
    return int(out.value)


def jb_dequantize_grad(q: int, qscale: float = 1.0) -> float:
    out = ctypes.c_float()
    _check(lib().jb_dequantize_grad(int(q), float(qscale), ctypes.byref(out)))
    return float(out.value)


def jb_max_seeds_per_call() -> int:
    return int(lib().jb_max_seeds_per_call())


# --- test hooks ---------------------------------------------------------------

def jb_debug_philox(seed, first_block: int, n_blocks: int, out, stream=None) -> None:
    """out: CUDA int32/uint32 tensor of >= 4 n_blocks words, 16-byte aligned."""
    _check(lib().jb_debug_philox(_seed(seed), int(first_block), int(n_blocks), out.data_ptr(),
                                 _stream(stream)))


def jb_debug_philox_fold(seed, first_block: int, n_blocks: int, out, stream=None) -> None:
    """out: CUDA int32/uint32 tensor of >= 1 element; receives the XOR of all words."""
    _check(lib().jb_debug_philox_fold(_seed(seed), int(first_block), int(n_blocks),
                                      out.data_ptr(), _stream(stream)))


def jb_debug_gaussian(seed, first_elem: int, n: int, out, stream=None) -> None:
    """out: CUDA float32 tensor of >= n elements."""
    _check(lib().jb_debug_gaussian(_seed(seed), int(first_elem), int(n), out.data_ptr(),
                                   _stream(stream)))


def jb_debug_box_muller(words, n_pairs: int, out, stream=None) -> None:
    """words: CUDA int32 tensor of 2 n_pairs words; out: float32 tensor of 2 n_pairs."""
    _check(lib().jb_debug_box_muller(words.data_ptr(), int(n_pairs), out.data_ptr(),
                                     _stream(stream)))


__all__ = [
    "JB_OK", "JB_F32", "JB_BF16", "SEED_DTYPE", "JbError", "ParamTable", "jb_segment", "jb_seed",
    "lib", "seeds_array", "default_flat_offsets", "jb_perturb", "jb_apply_updates",
    "jb_apply_updates_from", "jb_replay_updates", "jb_checksum", "jb_perturb_q4", "jb_q4_levels",
    "Q4Table", "jb_q4_segment",
    "jb_quantize_grad", "jb_dequantize_grad", "jb_max_seeds_per_call", "jb_status_string",
    "jb_debug_philox", "jb_debug_gaussian", "jb_debug_box_muller",
]
