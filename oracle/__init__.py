"""CPU oracle for the seeded-perturbation hot path (test infrastructure only).

Only the tests, ``__graft_entry__.smoke()`` and the CPU-baseline legs of
``bench.py`` import this package. It wraps ``jb_oracle.c`` (plain C, double
precision) with ctypes and numpy; it shares no code with the CUDA library and
never imports it. bf16 arrays are passed as numpy ``uint16`` bit patterns.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "jb_oracle.c")
_HDR = os.path.join(_HERE, "jb_oracle.h")
_OUT_DIR = os.path.join(_HERE, "_build")
_LIB = os.path.join(_OUT_DIR, "libjb_oracle.so")

F32, BF16 = 0, 1

SEED_DTYPE = np.dtype([("machine_id", "<u8"), ("step", "<u4"), ("sample_id", "<u4")])


class _Seed(ctypes.Structure):
    _fields_ = [("machine_id", ctypes.c_uint64), ("step", ctypes.c_uint32),
                ("sample_id", ctypes.c_uint32)]


_lock = threading.Lock()
_lib = None


def build(force: bool = False) -> str:
    """Compile the oracle with gcc (no fast-math, no contraction, OpenMP)."""
    os.makedirs(_OUT_DIR, exist_ok=True)
    stale = (not os.path.exists(_LIB) or
             max(os.path.getmtime(_SRC), os.path.getmtime(_HDR)) > os.path.getmtime(_LIB))
    if force or stale:
        tmp = _LIB + f".tmp{os.getpid()}"
        cmd = ["gcc", "-std=c11", "-O2", "-ffp-contract=off", "-fno-fast-math", "-fopenmp",
               "-fPIC", "-shared", "-D_GNU_SOURCE", _SRC, "-o", tmp, "-lm"]
        subprocess.run(cmd, check=True)
        os.replace(tmp, _LIB)
    return _LIB


def lib() -> ctypes.CDLL:
    global _lib
    with _lock:
        if _lib is None:
            path = build()
            L = ctypes.CDLL(path)
            vp = ctypes.c_void_p
            u32p = ctypes.POINTER(ctypes.c_uint32)
            u64 = ctypes.c_uint64
            L.jbo_philox4x32_10.argtypes = [u32p, u32p, u32p]
            L.jbo_block_words.argtypes = [_Seed, u64, u32p]
            L.jbo_philox_blocks.argtypes = [_Seed, u64, u64, vp]
            L.jbo_uniform_a.argtypes = [ctypes.c_uint32]
            L.jbo_uniform_a.restype = ctypes.c_double
            L.jbo_uniform_b.argtypes = [ctypes.c_uint32]
            L.jbo_uniform_b.restype = ctypes.c_double
            L.jbo_box_muller_pairs.argtypes = [vp, u64, vp]
            L.jbo_gaussian.argtypes = [_Seed, u64]
            L.jbo_gaussian.restype = ctypes.c_double
            L.jbo_gaussian_range.argtypes = [_Seed, u64, u64, vp]
            L.jbo_gaussian_at.argtypes = [_Seed, vp, u64, vp]
            L.jbo_round_bf16.argtypes = [ctypes.c_double]
            L.jbo_round_bf16.restype = ctypes.c_uint16
            L.jbo_bf16_to_double.argtypes = [ctypes.c_uint16]
            L.jbo_bf16_to_double.restype = ctypes.c_double
            L.jbo_perturb.argtypes = [vp, ctypes.c_int, u64, u64, _Seed, ctypes.c_double]
            L.jbo_perturb_at.argtypes = [vp, vp, ctypes.c_int, vp, u64, _Seed, ctypes.c_double]
            L.jbo_quantize.argtypes = [ctypes.c_double, ctypes.c_double]
            L.jbo_quantize.restype = ctypes.c_int8
            L.jbo_dequantize.argtypes = [ctypes.c_int8, ctypes.c_double]
            L.jbo_dequantize.restype = ctypes.c_double
            L.jbo_coefficient.argtypes = [ctypes.c_int8, ctypes.c_double, ctypes.c_double,
                                          ctypes.c_double]
            L.jbo_coefficient.restype = ctypes.c_float
            L.jbo_canonical_order.argtypes = [vp, ctypes.c_int, vp]
            L.jbo_canonical_order.restype = ctypes.c_int
            L.jbo_update.argtypes = [vp, ctypes.c_int, u64, u64, vp, vp, ctypes.c_int,
                                     ctypes.c_double, ctypes.c_double, ctypes.c_double]
            L.jbo_update.restype = ctypes.c_int
            L.jbo_update_at.argtypes = [vp, vp, ctypes.c_int, vp, u64, vp, vp, ctypes.c_int,
                                        ctypes.c_double, ctypes.c_double, ctypes.c_double]
            L.jbo_update_at.restype = ctypes.c_int
            L.jbo_update_delta_at.argtypes = [vp, u64, vp, vp, ctypes.c_int, ctypes.c_double,
                                              ctypes.c_double, ctypes.c_double, vp]
            L.jbo_update_delta_at.restype = ctypes.c_int
            L.jbo_update_delta_abs_at.argtypes = [vp, u64, vp, vp, ctypes.c_int, ctypes.c_double,
                                                  ctypes.c_double, ctypes.c_double, vp, vp]
            L.jbo_update_delta_abs_at.restype = ctypes.c_int
            L.jbo_q4_levels.argtypes = [vp]
            L.jbo_q4_quantize.argtypes = [vp, u64, vp, vp]
            L.jbo_q4_dequantize.argtypes = [vp, vp, u64, vp]
            L.jbo_q4_perturb.argtypes = [vp, vp, u64, u64, _Seed, ctypes.c_double, vp]
            L.jbo_q4_perturb.restype = ctypes.c_int
            L.jbo_window_hash.argtypes = [u64, u32p]
            L.jbo_window_hash.restype = ctypes.c_uint64
            L.jbo_checksum_segment.argtypes = [vp, ctypes.c_int, u64, u64]
            L.jbo_checksum_segment.restype = ctypes.c_uint64
            L.jbo_set_threads.argtypes = [ctypes.c_int]
            L.jbo_get_threads.restype = ctypes.c_int
            _lib = L
    return _lib


def _ptr(a: np.ndarray) -> ctypes.c_void_p:
    assert a.flags["C_CONTIGUOUS"]
    return ctypes.c_void_p(a.ctypes.data)


def _seed(s) -> _Seed:
    if isinstance(s, np.void) or (isinstance(s, np.ndarray) and s.dtype == SEED_DTYPE):
        return _Seed(int(s["machine_id"]), int(s["step"]), int(s["sample_id"]))
    mid, step, sample = s
    return _Seed(int(mid), int(step), int(sample))


def seeds_array(seeds) -> np.ndarray:
    """Seeds as a contiguous array of (machine_id, step, sample_id) records."""
    if isinstance(seeds, np.ndarray) and seeds.dtype == SEED_DTYPE:
        return np.ascontiguousarray(seeds)
    out = np.zeros(len(seeds), dtype=SEED_DTYPE)
    for i, (m, t, j) in enumerate(seeds):
        out[i] = (int(m), int(t), int(j))
    return out


def _dtype_code(a: np.ndarray) -> int:
    if a.dtype == np.float32:
        return F32
    if a.dtype == np.uint16:
        return BF16
    raise TypeError(f"oracle storage is float32 or uint16 (bf16 bits), got {a.dtype}")


# --- generator -------------------------------------------------------------

def philox(ctr, key) -> np.ndarray:
    c = (ctypes.c_uint32 * 4)(*[int(v) & 0xFFFFFFFF for v in ctr])
    k = (ctypes.c_uint32 * 2)(*[int(v) & 0xFFFFFFFF for v in key])
    o = (ctypes.c_uint32 * 4)()
    lib().jbo_philox4x32_10(c, k, o)
    return np.array(list(o), dtype=np.uint32)


def philox_blocks(seed, first_block: int, n_blocks: int) -> np.ndarray:
    out = np.empty((n_blocks, 4), dtype=np.uint32)
    lib().jbo_philox_blocks(_seed(seed), first_block, n_blocks, _ptr(out))
    return out


def uniform_a(x: int) -> float:
    return lib().jbo_uniform_a(int(x))


def uniform_b(x: int) -> float:
    return lib().jbo_uniform_b(int(x))


def box_muller_pairs(words: np.ndarray) -> np.ndarray:
    w = np.ascontiguousarray(words, dtype=np.uint32).reshape(-1, 2)
    out = np.empty(w.shape, dtype=np.float64)
    lib().jbo_box_muller_pairs(_ptr(w), w.shape[0], _ptr(out))
    return out


def gaussian(seed, e: int) -> float:
    return lib().jbo_gaussian(_seed(seed), int(e))


def gaussian_range(seed, first: int, n: int) -> np.ndarray:
    out = np.empty(n, dtype=np.float64)
    lib().jbo_gaussian_range(_seed(seed), first, n, _ptr(out))
    return out


def gaussian_at(seed, idx: np.ndarray) -> np.ndarray:
    i = np.ascontiguousarray(idx, dtype=np.uint64)
    out = np.empty(i.shape[0], dtype=np.float64)
    lib().jbo_gaussian_at(_seed(seed), _ptr(i), i.shape[0], _ptr(out))
    return out


# --- storage types ---------------------------------------------------------

def round_bf16(x) -> np.ndarray:
    xs = np.atleast_1d(np.asarray(x, dtype=np.float64))
    f = lib().jbo_round_bf16
    return np.array([f(float(v)) for v in xs], dtype=np.uint16)


def bf16_to_f64(h: np.ndarray) -> np.ndarray:
    h = np.ascontiguousarray(h, dtype=np.uint16)
    return (h.astype(np.uint32) << 16).view(np.float32).astype(np.float64)


# --- perturbation and update -----------------------------------------------

def perturb(theta: np.ndarray, flat_offset: int, seed, eps: float) -> np.ndarray:
    """Returns PerturbParameters applied to a copy of theta."""
    out = np.array(theta, copy=True, order="C")
    lib().jbo_perturb(_ptr(out), _dtype_code(out), out.size, flat_offset, _seed(seed), eps)
    return out


def perturb_at(values: np.ndarray, idx: np.ndarray, seed, eps: float) -> np.ndarray:
    v = np.ascontiguousarray(values)
    i = np.ascontiguousarray(idx, dtype=np.uint64)
    out = np.empty_like(v)
    lib().jbo_perturb_at(_ptr(v), _ptr(out), _dtype_code(v), _ptr(i), i.size, _seed(seed), eps)
    return out


def quantize(g: float, qscale: float = 1.0) -> int:
    return int(lib().jbo_quantize(float(g), float(qscale)))


def dequantize(q: int, qscale: float = 1.0) -> float:
    return float(lib().jbo_dequantize(int(q), float(qscale)))


def coefficient(q: int, lr: float, denom: float, qscale: float) -> float:
    return float(lib().jbo_coefficient(int(q), float(lr), float(denom), float(qscale)))


def canonical_order(seeds) -> np.ndarray:
    s = seeds_array(seeds)
    perm = np.empty(len(s), dtype=np.int32)
    rc = lib().jbo_canonical_order(_ptr(s), len(s), _ptr(perm))
    if rc != 0:
        raise ValueError("duplicate seed")
    return perm


def _check(rc: int):
    if rc == -1:
        raise ValueError("duplicate seed")
    if rc != 0:
        raise MemoryError("oracle allocation failed")


def update(theta: np.ndarray, flat_offset: int, seeds, q, lr: float, denom: float,
           qscale: float) -> np.ndarray:
    """Returns the step update applied to a copy of theta."""
    out = np.array(theta, copy=True, order="C")
    s = seeds_array(seeds)
    qa = np.ascontiguousarray(q, dtype=np.int8)
    _check(lib().jbo_update(_ptr(out), _dtype_code(out), out.size, flat_offset, _ptr(s),
                            _ptr(qa), len(s), lr, denom, qscale))
    return out


def update_at(values: np.ndarray, idx: np.ndarray, seeds, q, lr: float, denom: float,
              qscale: float) -> np.ndarray:
    v = np.ascontiguousarray(values)
    i = np.ascontiguousarray(idx, dtype=np.uint64)
    s = seeds_array(seeds)
    qa = np.ascontiguousarray(q, dtype=np.int8)
    out = np.empty_like(v)
    _check(lib().jbo_update_at(_ptr(v), _ptr(out), _dtype_code(v), _ptr(i), i.size, _ptr(s),
                               _ptr(qa), len(s), lr, denom, qscale))
    return out


def update_delta_at(idx: np.ndarray, seeds, q, lr: float, denom: float,
                    qscale: float) -> np.ndarray:
    i = np.ascontiguousarray(idx, dtype=np.uint64)
    s = seeds_array(seeds)
    qa = np.ascontiguousarray(q, dtype=np.int8)
    out = np.empty(i.size, dtype=np.float64)
    _check(lib().jbo_update_delta_at(_ptr(i), i.size, _ptr(s), _ptr(qa), len(s), lr, denom,
                                     qscale, _ptr(out)))
    return out


def update_delta_abs_at(idx: np.ndarray, seeds, q, lr: float, denom: float,
                        qscale: float) -> tuple:
    """(sum_k c_k z_k, sum_k |c_k z_k|) at global indices idx, in double; the first
    is update_delta_at's value bit for bit."""
    i = np.ascontiguousarray(idx, dtype=np.uint64)
    s = seeds_array(seeds)
    qa = np.ascontiguousarray(q, dtype=np.int8)
    out = np.empty(i.size, dtype=np.float64)
    mag = np.empty(i.size, dtype=np.float64)
    _check(lib().jbo_update_delta_abs_at(_ptr(i), i.size, _ptr(s), _ptr(qa), len(s), lr, denom,
                                         qscale, _ptr(out), _ptr(mag)))
    return out, mag


# --- 4-bit weights -----------------------------------------------------------

def q4_levels() -> np.ndarray:
    out = np.empty(16, dtype=np.float32)
    lib().jbo_q4_levels(_ptr(out))
    return out


def q4_quantize(w) -> tuple:
    """(codes uint8[(n + 1) // 2], scales float32[ceil(n / 64)]) of values w."""
    w = np.ascontiguousarray(w, dtype=np.float64)
    codes = np.zeros((w.size + 1) // 2, dtype=np.uint8)
    scale = np.zeros((w.size + 63) // 64, dtype=np.float32)
    lib().jbo_q4_quantize(_ptr(w), w.size, _ptr(codes), _ptr(scale))
    return codes, scale


def q4_dequantize(codes, scale, n: int) -> np.ndarray:
    codes = np.ascontiguousarray(codes, dtype=np.uint8)
    scale = np.ascontiguousarray(scale, dtype=np.float32)
    w = np.empty(n, dtype=np.float64)
    lib().jbo_q4_dequantize(_ptr(codes), _ptr(scale), n, _ptr(w))
    return w


def q4_perturb(codes, scale, n: int, flat_offset: int, seed, eps: float):
    """(codes', scales', perturbed values before quantization) of one 4-bit tensor."""
    c = np.array(codes, dtype=np.uint8, copy=True)
    s = np.array(scale, dtype=np.float32, copy=True)
    w = np.empty(n, dtype=np.float64)
    _check(lib().jbo_q4_perturb(_ptr(c), _ptr(s), n, flat_offset, _seed(seed), eps, _ptr(w)))
    return c, s, w


# --- model checksum ----------------------------------------------------------

def window_hash(window: int, words) -> int:
    w = (ctypes.c_uint32 * 4)(*[int(x) & 0xFFFFFFFF for x in words])
    return int(lib().jbo_window_hash(int(window), w))


def checksum(tensors, flat_offsets) -> int:
    """Sum mod 2^64 of the per-segment window contributions (see jb_oracle.c)."""
    total = 0
    for t, fo in zip(tensors, flat_offsets):
        a = np.ascontiguousarray(t)
        total += int(lib().jbo_checksum_segment(_ptr(a), _dtype_code(a), a.size, int(fo)))
    return total % (1 << 64)


def set_threads(n: int) -> None:
    lib().jbo_set_threads(int(n))


def get_threads() -> int:
    return int(lib().jbo_get_threads())
