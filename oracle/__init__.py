"""CPU oracle of the committed AdamW step and its bit-exact state digest.

TEST INFRASTRUCTURE ONLY: the tests, ``__graft_entry__.smoke()`` and the
benchmark's ``cpu_baseline`` / ``--impl reference`` legs are the only callers.
The library path never imports this package, and this package never imports
the library.  The arithmetic is in ``apc_oracle.c`` (plain C, gcc
``-O2 -ffp-contract=off``); this module builds it and wraps it with ctypes.

Definitions (arxiv 2609.18178, Section III-A Eq. 2 for the preserved state
W, M, V, tau_opt; Section I and III-C phase 2 for the committed boundary;
Abstract and Section IV-F/IV-G for the bitwise state checks):

* ``resolve_hparams``: the eight binary32 scalars of step t, each formed in
  double from the decimal hyper-parameters and rounded once.
* ``commit``: AdamW in place over one tensor in the fixed binary32 order,
  bf16 round-to-nearest-even copy of p', and the four digests
  ``sum_i splitmix64(((G_i mod 2^32) << 32) | bits(i)) mod 2^64`` of
  p', m', v' and the bf16 copy.
* ``commit_bf16``: the same step with p, m, v stored in bf16 (Section IV-A
  keeps parameters and moments in BF16): widened exactly, updated in the
  same order, each rounded once to bf16; digests of p', m', v'.
* ``count_nonzero``: the quiescence guard's count of nonzero words
  (Section III-C, phase 2).
"""
from __future__ import annotations

import ctypes
import fcntl
import os
import platform
import subprocess

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_BUILD = os.path.join(_HERE, "_build", platform.machine())
_SO = os.path.join(_BUILD, "liboracle.so")
_SRC = os.path.join(_HERE, "apc_oracle.c")

MASK64 = (1 << 64) - 1
# order of the resolved scalars
HB1, HOMB1, HB2, HOMB2, HEPS, HDECAY, HSTEP, HRSB2 = range(8)


def build() -> str:
    """Compile liboracle.so (plain C) if it is missing or stale."""
    os.makedirs(_BUILD, exist_ok=True)
    with open(os.path.join(_BUILD, ".lock"), "w") as lk:
        fcntl.flock(lk, fcntl.LOCK_EX)
        if os.path.exists(_SO) and os.path.getmtime(_SO) >= os.path.getmtime(_SRC):
            return _SO
        tmp = _SO + ".tmp%d" % os.getpid()
        subprocess.run(["gcc", "-O2", "-std=c11", "-ffp-contract=off", "-fno-fast-math", "-fPIC", "-shared",
                        "-pthread", "-fvisibility=hidden", _SRC, "-o", tmp, "-lm"], check=True)
        os.replace(tmp, _SO)
    return _SO


_lib = None


def _L():
    global _lib
    if _lib is None:
        lib = ctypes.CDLL(build())
        vp, u64, i64, d = ctypes.c_void_p, ctypes.c_uint64, ctypes.c_int64, ctypes.c_double
        lib.oracle_resolve_hparams.argtypes = [d, d, d, d, d, i64, vp]
        lib.oracle_resolve_hparams.restype = ctypes.c_int
        lib.oracle_adamw.argtypes = [vp, vp, vp, vp, vp, u64, vp]
        lib.oracle_adamw.restype = None
        lib.oracle_splitmix64.argtypes = [u64]
        lib.oracle_splitmix64.restype = u64
        lib.oracle_digest_u32.argtypes = [vp, u64, u64]
        lib.oracle_digest_u32.restype = u64
        lib.oracle_digest_u16.argtypes = [vp, u64, u64]
        lib.oracle_digest_u16.restype = u64
        lib.oracle_bf16_rne.argtypes = [ctypes.c_float]
        lib.oracle_bf16_rne.restype = ctypes.c_uint16
        lib.oracle_bf16_rne_array.argtypes = [vp, vp, u64]
        lib.oracle_bf16_rne_array.restype = None
        lib.oracle_commit.argtypes = [vp, vp, vp, vp, vp, u64, u64, vp, vp]
        lib.oracle_commit.restype = None
        lib.oracle_commit_mt.argtypes = [vp, vp, vp, vp, vp, u64, u64, vp, vp, ctypes.c_int]
        lib.oracle_commit_mt.restype = None
        lib.oracle_adamw_bf16.argtypes = [vp, vp, vp, vp, u64, vp]
        lib.oracle_adamw_bf16.restype = None
        lib.oracle_commit_bf16.argtypes = [vp, vp, vp, vp, u64, u64, vp, vp]
        lib.oracle_commit_bf16.restype = None
        lib.oracle_count_nonzero_u16.argtypes = [vp, u64]
        lib.oracle_count_nonzero_u16.restype = u64
        lib.oracle_count_nonzero_u32.argtypes = [vp, u64]
        lib.oracle_count_nonzero_u32.restype = u64
        _lib = lib
    return _lib


DEFAULT_HP = dict(lr=3e-4, beta1=0.9, beta2=0.95, eps=1e-8, weight_decay=0.1)


def resolve_hparams(hp: dict, step: int) -> np.ndarray:
    """The eight binary32 scalars (b1, 1-b1, b2, 1-b2, eps, 1-lr*wd,
    lr/(1-b1^t), 1/sqrt(1-b2^t)) of step ``step``."""
    out = np.zeros(8, dtype=np.float32)
    rc = _L().oracle_resolve_hparams(hp["lr"], hp["beta1"], hp["beta2"], hp["eps"], hp["weight_decay"],
                                     int(step), out.ctypes.data)
    if rc != 0:
        raise ValueError("hyper-parameters out of range")
    return out


def _c(a, dt):
    assert a.dtype == dt and a.flags.c_contiguous, (a.dtype, dt)
    return a.ctypes.data


def adamw(p, m, v, g, h8) -> np.ndarray:
    """AdamW in place on float32 p, m, v with uint16 bf16 grad g; returns the
    uint16 bf16 copy of p'."""
    n = p.size
    assert m.size == n and v.size == n and g.size == n
    w = np.empty(n, dtype=np.uint16)
    _L().oracle_adamw(_c(p, np.float32), _c(m, np.float32), _c(v, np.float32), _c(g, np.uint16), w.ctypes.data,
                      n, _c(np.ascontiguousarray(h8, dtype=np.float32), np.float32))
    return w


def splitmix64(x: int) -> int:
    return int(_L().oracle_splitmix64(int(x) & MASK64))


def digest_f32(a: np.ndarray, goff: int = 0) -> int:
    """Digest of a float32 (or uint32 bits) array at global offset goff."""
    a = np.ascontiguousarray(a)
    assert a.dtype in (np.float32, np.uint32)
    return int(_L().oracle_digest_u32(a.ctypes.data, a.size, int(goff) & MASK64))


def digest_u16(a: np.ndarray, goff: int = 0) -> int:
    """Digest of a uint16 (bf16 bits) array at global offset goff."""
    a = np.ascontiguousarray(a, dtype=np.uint16)
    return int(_L().oracle_digest_u16(a.ctypes.data, a.size, int(goff) & MASK64))


def bf16_rne(x: np.ndarray) -> np.ndarray:
    x = np.ascontiguousarray(x, dtype=np.float32)
    out = np.empty(x.size, dtype=np.uint16)
    _L().oracle_bf16_rne_array(x.ctypes.data, out.ctypes.data, x.size)
    return out.reshape(x.shape)


def commit(p, m, v, g, goff: int, h8, nthreads: int = 1):
    """Committed step over one tensor, in place.  Returns (w, [Dp, Dm, Dv, Dw])."""
    n = p.size
    assert m.size == n and v.size == n and g.size == n
    w = np.empty(n, dtype=np.uint16)
    d = np.zeros(4, dtype=np.uint64)
    h = np.ascontiguousarray(h8, dtype=np.float32)
    args = (_c(p, np.float32), _c(m, np.float32), _c(v, np.float32), _c(g, np.uint16), w.ctypes.data, n,
            int(goff) & MASK64, h.ctypes.data, d.ctypes.data)
    if nthreads > 1:
        _L().oracle_commit_mt(*args, int(nthreads))
    else:
        _L().oracle_commit(*args)
    return w, [int(x) for x in d]


def adamw_bf16(p, m, v, g, h8) -> None:
    """bf16-state AdamW in place on uint16 p, m, v with uint16 grad g."""
    n = p.size
    assert m.size == n and v.size == n and g.size == n
    _L().oracle_adamw_bf16(_c(p, np.uint16), _c(m, np.uint16), _c(v, np.uint16), _c(g, np.uint16), n,
                           _c(np.ascontiguousarray(h8, dtype=np.float32), np.float32))


def commit_bf16(p, m, v, g, goff: int, h8):
    """bf16-state committed step over one tensor, in place.  Returns the three
    digests [Dp', Dm', Dv'] of the written bf16 words."""
    n = p.size
    assert m.size == n and v.size == n and g.size == n
    d = np.zeros(3, dtype=np.uint64)
    h = np.ascontiguousarray(h8, dtype=np.float32)
    _L().oracle_commit_bf16(_c(p, np.uint16), _c(m, np.uint16), _c(v, np.uint16), _c(g, np.uint16), n,
                            int(goff) & MASK64, h.ctypes.data, d.ctypes.data)
    return [int(x) for x in d]


def count_nonzero(a: np.ndarray) -> int:
    """Words of a uint16/float32/uint32 array whose bit pattern is nonzero."""
    a = np.ascontiguousarray(a)
    if a.dtype == np.uint16:
        return int(_L().oracle_count_nonzero_u16(a.ctypes.data, a.size))
    assert a.dtype in (np.float32, np.uint32)
    return int(_L().oracle_count_nonzero_u32(a.ctypes.data, a.size))


def commit_table(tensors, h8, nthreads: int = 1):
    """Committed step over a chunk table: ``tensors`` is a list of dicts with
    float32 p, m, v, uint16 g and int goff.  Returns (list of w, 4 digests)."""
    ws, tot = [], [0, 0, 0, 0]
    for t in tensors:
        w, d = commit(t["p"], t["m"], t["v"], t["g"], t["goff"], h8, nthreads)
        ws.append(w)
        tot = [(a + b) & MASK64 for a, b in zip(tot, d)]
    return ws, tot
