"""CPU oracle of the KronQ per-layer quantization path.

TEST INFRASTRUCTURE ONLY: imported by tests/, by __graft_entry__.smoke() and by the
benchmark's CPU-baseline leg. The CUDA library never imports, links or runs it, and the
two share no code.

  kronq_oracle  float64 statement of every step (numpy)
  sweep32.c     the fp32-ordered OBS sweep (plain C, -ffp-contract=off, OpenMP over rows)
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import sys

import numpy as np

from . import kronq_oracle as ref  # noqa: F401

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "sweep32.c")
_LIB = os.path.join(_HERE, "_build", "libkqref_sweep32.so")
_lib = None


def build(force: bool = False) -> str:
    """Compile sweep32.c into oracle/_build/libkqref_sweep32.so (gcc, portable flags)."""
    os.makedirs(os.path.dirname(_LIB), exist_ok=True)
    if not force and os.path.exists(_LIB) and os.path.getmtime(_LIB) >= os.path.getmtime(_SRC):
        return _LIB
    cmd = ["gcc", "-O2", "-std=c11", "-ffp-contract=off", "-fno-fast-math", "-fPIC", "-shared",
           "-fopenmp", _SRC, "-o", _LIB + ".tmp", "-lm"]
    subprocess.run(cmd, check=True)
    os.replace(_LIB + ".tmp", _LIB)
    return _LIB


def _load():
    global _lib
    if _lib is None:
        lib = ctypes.CDLL(build())
        f = lib.kqref_sweep32
        P = ctypes.c_void_p
        I64 = ctypes.c_int64
        f.argtypes = [P, I64, I64, P, P, ctypes.c_int, ctypes.c_int, ctypes.c_int, P, I64,
                      P, P, P, P, P]
        f.restype = ctypes.c_int
        _lib = lib
    return _lib


def obs_sweep_fp32(W, Lt, bits: int, group: int, block: int = 128, rows=None,
                   want_pre_q: bool = False, Pt=None) -> dict:
    """fp32-ordered sweep of Algorithm 2 (see sweep32.c) on float32 W [m, n] and
    Lt = R^T [n, n]; with the GPTAQ correction when Pt = P^T [n, n] is given. `rows`
    selects a subset of rows (all rows by default)."""
    W = np.ascontiguousarray(W, dtype=np.float32)
    Lt = np.ascontiguousarray(Lt, dtype=np.float32)
    m, n = W.shape
    assert Lt.shape == (n, n)
    if Pt is not None:
        Pt = np.ascontiguousarray(Pt, dtype=np.float32)
        assert Pt.shape == (n, n)
    if rows is None:
        rows_arr = None
        nrows = m
    else:
        rows_arr = np.ascontiguousarray(rows, dtype=np.int64)
        nrows = rows_arr.shape[0]
    ng = 1 if group == 0 else (n + group - 1) // group
    codes = np.zeros((nrows, n), np.uint8)
    scale = np.zeros((nrows, ng), np.float32)
    zero = np.zeros((nrows, ng), np.float32)
    E = np.zeros((nrows, n), np.float32)
    pre_q = np.zeros((nrows, n), np.float32) if want_pre_q else None
    ptr = lambda a: None if a is None else a.ctypes.data  # noqa: E731
    rc = _load().kqref_sweep32(ptr(W), m, n, ptr(Lt), ptr(Pt), bits, group, block, ptr(rows_arr), nrows,
                               ptr(codes), ptr(scale), ptr(zero), ptr(E), ptr(pre_q))
    if rc != 0:
        raise ValueError("kqref_sweep32 rejected its arguments")
    out = {"codes": codes, "scale": scale, "zero": zero, "E": E}
    if want_pre_q:
        out["pre_q"] = pre_q
    return out


if __name__ == "__main__":
    print(build(force="--force" in sys.argv))
