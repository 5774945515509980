import os
import subprocess
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

BUILD = os.path.join(ROOT, "tests", "_build")


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a CUDA GPU (GB300, sm_103a)")
    config.addinivalue_line("markers", "slow: long-running CPU check")


@pytest.fixture(scope="session")
def aten_philox():
    """ctypes handle on a tiny library that calls at::Philox4_32."""
    import ctypes
    import torch
    os.makedirs(BUILD, exist_ok=True)
    src = os.path.join(ROOT, "tests", "helpers", "aten_philox.cpp")
    out = os.path.join(BUILD, "libaten_philox.so")
    if not os.path.exists(out) or os.path.getmtime(src) > os.path.getmtime(out):
        inc = os.path.join(os.path.dirname(torch.__file__), "include")
        tmp = out + f".tmp{os.getpid()}"
        subprocess.run(["g++", "-std=c++17", "-O1", "-fPIC", "-shared", "-I", inc, src,
                        "-o", tmp], check=True)
        os.replace(tmp, out)
    L = ctypes.CDLL(out)
    L.aten_philox_blocks.argtypes = [ctypes.c_uint64] * 4 + [ctypes.c_void_p]
    L.aten_philox_rounds.argtypes = [ctypes.c_uint64] * 3 + [ctypes.c_int, ctypes.c_void_p]
    return L


@pytest.fixture(scope="session")
def oracle_lib():
    import oracle
    oracle.lib()
    return oracle
