"""Seeded synthetic inputs for the committed-step workloads.

The value recipe lives in ``philox.h`` (Philox4x32-10 random bits, an
Irwin-Hall normal, the per-buffer scalings of the fp32 master parameters,
moments and bf16 gradient).  This module builds the host fill library
(``libsynth_host.so``, gcc) and the device fill library (``libsynth_dev.so``,
nvcc for sm_103a) and wraps both with ctypes.  It serves the tests, the bench
and the CPU oracle's callers alike, and holds none of the committed step's own
arithmetic.
"""
from __future__ import annotations

import ctypes
import fcntl
import os
import platform
import subprocess

import numpy as np

P, M, V, G = 1, 2, 3, 4
GZERO = 5
P16, M16, V16 = 6, 7, 8
SEED = 0

_HERE = os.path.dirname(os.path.abspath(__file__))
_BUILD = os.path.join(_HERE, "_build", platform.machine())
_HOST_SO = os.path.join(_BUILD, "libsynth_host.so")
_DEV_SO = os.path.join(_BUILD, "libsynth_dev.so")
_SRC_H = os.path.join(_HERE, "philox.h")
_SRC_HOST = os.path.join(_HERE, "synth_host.c")
_SRC_DEV = os.path.join(_HERE, "synth_dev.cu")


def _stale(target: str, sources: list[str]) -> bool:
    if not os.path.exists(target):
        return True
    t = os.path.getmtime(target)
    return any(os.path.getmtime(s) > t for s in sources)


def _locked_build(target: str, sources: list[str], cmd_for) -> None:
    os.makedirs(_BUILD, exist_ok=True)
    with open(os.path.join(_BUILD, ".lock"), "w") as lk:
        fcntl.flock(lk, fcntl.LOCK_EX)
        if not _stale(target, sources):
            return
        tmp = target + ".tmp%d" % os.getpid()
        subprocess.run(cmd_for(tmp), check=True)
        os.replace(tmp, target)


def build_host() -> str:
    _locked_build(_HOST_SO, [_SRC_H, _SRC_HOST], lambda out: [
        "gcc", "-O3", "-std=c11", "-ffp-contract=off", "-fno-fast-math", "-fPIC", "-shared",
        "-pthread", "-fvisibility=hidden", _SRC_HOST, "-o", out])
    return _HOST_SO


def build_dev() -> str:
    nvcc = os.environ.get("NVCC", "nvcc")
    _locked_build(_DEV_SO, [_SRC_H, _SRC_DEV], lambda out: [
        nvcc, "-gencode", "arch=compute_103a,code=sm_103a", "-O3", "-lineinfo", "-fmad=false",
        "-Xcompiler", "-fPIC,-fvisibility=hidden", "-shared", _SRC_DEV, "-o", out])
    return _DEV_SO


_host = None
_dev = None


def _host_lib():
    global _host
    if _host is None:
        lib = ctypes.CDLL(build_host())
        lib.synth_fill.argtypes = [ctypes.c_int, ctypes.c_uint64, ctypes.c_uint64, ctypes.c_uint64,
                                   ctypes.c_int64, ctypes.c_void_p, ctypes.c_int]
        lib.synth_fill.restype = ctypes.c_int
        lib.synth_fill_at.argtypes = [ctypes.c_int, ctypes.c_uint64, ctypes.c_void_p, ctypes.c_uint64,
                                      ctypes.c_int64, ctypes.c_void_p]
        lib.synth_fill_at.restype = ctypes.c_int
        lib.synth_philox.argtypes = [ctypes.c_void_p, ctypes.c_uint32, ctypes.c_uint32, ctypes.c_void_p]
        lib.synth_philox.restype = None
        lib.synth_normal_at.argtypes = [ctypes.c_uint64, ctypes.c_int, ctypes.c_uint64, ctypes.c_int64]
        lib.synth_normal_at.restype = ctypes.c_double
        _host = lib
    return _host


def _dev_lib():
    global _dev
    if _dev is None:
        lib = ctypes.CDLL(build_dev())
        lib.synth_fill_dev.argtypes = [ctypes.c_int, ctypes.c_uint64, ctypes.c_uint64, ctypes.c_uint64,
                                       ctypes.c_int64, ctypes.c_void_p, ctypes.c_void_p]
        lib.synth_fill_dev.restype = ctypes.c_int
        _dev = lib
    return _dev


def _dtype(kind: int):
    if kind in (P, M, V):
        return np.float32
    if kind in (G, P16, M16, V16):
        return np.uint16
    raise ValueError("unknown synthetic buffer kind %r" % (kind,))


def fill(kind: int, n: int, goff: int = 0, step: int = 0, seed: int = SEED,
         nthreads: int | None = None, out: np.ndarray | None = None) -> np.ndarray:
    """Values of global indices goff..goff+n-1 as a numpy array (float32, or
    uint16 bf16 bits for the gradient)."""
    dt = _dtype(kind)
    if out is None:
        out = np.empty(n, dtype=dt)
    assert out.dtype == dt and out.size == n and out.flags.c_contiguous
    if nthreads is None:
        nthreads = os.cpu_count() or 1
    rc = _host_lib().synth_fill(kind, seed, goff, n, step, out.ctypes.data, nthreads)
    if rc != 0:
        raise RuntimeError("synth_fill failed (%d)" % rc)
    return out


def fill_at(kind: int, idx, step: int = 0, seed: int = SEED) -> np.ndarray:
    """Values at arbitrary global indices."""
    idx = np.ascontiguousarray(idx, dtype=np.uint64)
    out = np.empty(idx.size, dtype=_dtype(kind))
    rc = _host_lib().synth_fill_at(kind, seed, idx.ctypes.data, idx.size, step, out.ctypes.data)
    if rc != 0:
        raise RuntimeError("synth_fill_at failed (%d)" % rc)
    return out


def fill_dev(kind: int, ptr: int, n: int, goff: int = 0, step: int = 0, seed: int = SEED,
             stream: int = 0) -> None:
    """Fill a device buffer at address ``ptr`` (n elements) on ``stream``."""
    _dtype(kind)
    rc = _dev_lib().synth_fill_dev(kind, seed, goff, n, step, ctypes.c_void_p(ptr), ctypes.c_void_p(stream))
    if rc != 0:
        raise RuntimeError("synth_fill_dev failed (cuda error %d)" % rc)


def philox(ctr, key) -> list[int]:
    """One raw Philox4x32-10 block (for known-answer tests)."""
    c = (ctypes.c_uint32 * 4)(*[int(x) & 0xFFFFFFFF for x in ctr])
    o = (ctypes.c_uint32 * 4)()
    _host_lib().synth_philox(ctypes.addressof(c), int(key[0]) & 0xFFFFFFFF, int(key[1]) & 0xFFFFFFFF,
                             ctypes.addressof(o))
    return list(o)


def normal_at(kind: int, i: int, step: int = 0, seed: int = SEED) -> float:
    return _host_lib().synth_normal_at(seed, kind, i, step)


def state(n: int, goff: int = 0, seed: int = SEED, nthreads: int | None = None):
    """(p, m, v) fp32 state arrays of one contiguous global range."""
    return (fill(P, n, goff, 0, seed, nthreads), fill(M, n, goff, 0, seed, nthreads),
            fill(V, n, goff, 0, seed, nthreads))


def state_bf16(n: int, goff: int = 0, seed: int = SEED, nthreads: int | None = None):
    """(p, m, v) bf16 state bits (uint16) of one contiguous global range."""
    return (fill(P16, n, goff, 0, seed, nthreads), fill(M16, n, goff, 0, seed, nthreads),
            fill(V16, n, goff, 0, seed, nthreads))


def grad(n: int, goff: int = 0, step: int = 1, seed: int = SEED, nthreads: int | None = None):
    """bf16 gradient bits (uint16) of one contiguous global range for step ``step``."""
    return fill(G, n, goff, step, seed, nthreads)
