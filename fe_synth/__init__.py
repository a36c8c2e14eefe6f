"""Seeded synthetic inputs for the cascaded drafter (tests and benchmark).

This module draws numbers and lays them out; it computes nothing of the drafter.
The C generator (``synth.c``) is a pure function of (seed, tensor_id, index), so the
oracle and the CUDA path receive byte-identical inputs. ``workloads.py`` holds the
named workload shapes and the recipe that turns them into host tensors.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "synth.c")
_LIB = os.path.join(_HERE, "libfe_synth.so")
_lock = threading.Lock()
_lib = None


def build(force: bool = False) -> str:
    """Compile synth.c into libfe_synth.so (portable flags only)."""
    if force or not os.path.exists(_LIB) or os.path.getmtime(_LIB) < os.path.getmtime(_SRC):
        tmp = _LIB + f".tmp{os.getpid()}"
        subprocess.check_call(["gcc", "-O2", "-std=c99", "-fPIC", "-shared", "-fopenmp",
                               "-ffp-contract=off", _SRC, "-o", tmp])
        os.replace(tmp, _LIB)
    return _LIB


def lib():
    global _lib
    with _lock:
        if _lib is None:
            build()
            L = ctypes.CDLL(_LIB)
            L.synth_fill_normal.argtypes = [ctypes.c_uint64, ctypes.c_uint64, ctypes.c_int64,
                                            ctypes.c_double, ctypes.c_int32, ctypes.c_void_p]
            L.synth_fill_normal_slice.argtypes = [ctypes.c_uint64, ctypes.c_uint64, ctypes.c_int64,
                                                  ctypes.c_int64, ctypes.c_double, ctypes.c_int32,
                                                  ctypes.c_void_p]
            L.synth_fill_uniform_int.argtypes = [ctypes.c_uint64, ctypes.c_uint64, ctypes.c_int64,
                                                 ctypes.c_int64, ctypes.c_int64, ctypes.c_void_p]
            L.synth_permutation.argtypes = [ctypes.c_uint64, ctypes.c_uint64, ctypes.c_int64,
                                            ctypes.c_void_p]
            L.synth_splitmix64.argtypes = [ctypes.c_uint64]
            L.synth_splitmix64.restype = ctypes.c_uint64
            _lib = L
    return _lib


def fill_normal(t, seed: int, tensor_id: int, std: float) -> None:
    """Fill a contiguous CPU torch tensor (float32 or bfloat16) with N(0, std^2) deviates."""
    import torch
    assert t.device.type == "cpu" and t.is_contiguous()
    dt = {torch.float32: 0, torch.bfloat16: 1}[t.dtype]
    lib().synth_fill_normal(seed, tensor_id, t.numel(), std, dt, t.data_ptr())


def fill_uniform_int(t, seed: int, tensor_id: int, lo: int, hi: int) -> None:
    """Fill a contiguous CPU int32 tensor with integers uniform in [lo, hi]."""
    import torch
    assert t.device.type == "cpu" and t.is_contiguous() and t.dtype == torch.int32
    lib().synth_fill_uniform_int(seed, tensor_id, t.numel(), lo, hi, t.data_ptr())


def permutation(t, seed: int, tensor_id: int) -> None:
    import torch
    assert t.device.type == "cpu" and t.is_contiguous() and t.dtype == torch.int32
    lib().synth_permutation(seed, tensor_id, t.numel(), t.data_ptr())


def splitmix64(z: int) -> int:
    return int(lib().synth_splitmix64(z))
