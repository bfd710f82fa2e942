"""In-tree build of libapc.so for sm_103a (nvcc, no cmake).

The translation units compile in parallel; the result lands in
``paper_2609_18178_gb300/_build/<machine>/libapc.so`` (git-ignored), next to
the sources, so a GPU host builds its own copy for its own architecture.
"""
from __future__ import annotations

import fcntl
import hashlib
import os
import platform
import subprocess

HERE = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(HERE)
CSRC = os.path.join(HERE, "csrc")
INCLUDE = os.path.join(ROOT, "include")
BUILD = os.path.join(HERE, "_build", platform.machine())
# APC_BUILD_DEFINES (read at import), e.g. "-DAPC_COMMIT_CONSUMER_WARPS=11
# -DAPC_SMEM_CARVEOUT=100", builds and loads a variant of the library with
# other compile-time kernel shapes (the APC_* macros of csrc/apc_internal.h),
# in a folder of its own, for shape experiments; unset, the default build.
DEFINES = os.environ.get("APC_BUILD_DEFINES", "").split()
for _d in DEFINES:
    if not _d.startswith("-DAPC_"):
        raise ValueError("APC_BUILD_DEFINES takes -DAPC_... macro definitions only, got %r" % _d)
LIB_DIR = (os.path.join(BUILD, "variant-" + hashlib.sha1(" ".join(DEFINES).encode()).hexdigest()[:12])
           if DEFINES else BUILD)
LIB = os.path.join(LIB_DIR, "libapc.so")

ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]
# exact IEEE binary32: no contraction into FMA, IEEE divide and sqrt, denormals kept
NUMERIC = ["-fmad=false", "-prec-div=true", "-prec-sqrt=true", "-ftz=false"]
UNITS = ["apc_commit.cu", "apc_digest.cu", "apc_guard.cu", "apc_upload.cu", "apc_host.cpp"]
# The integer-pipe probe is a library of its own: the benchmark's
# measurement tool for the verification pass's roofline, not the hot path.
PROBE_LIB = os.path.join(BUILD, "libapc_probe.so")
PROBE_SRC = os.path.join(CSRC, "apc_probe.cu")


def sources() -> list[str]:
    out = [os.path.join(CSRC, u) for u in UNITS]
    out += [os.path.join(CSRC, h) for h in ("apc_internal.h", "apc_device.cuh", "apc_tma.cuh")]
    out.append(os.path.join(INCLUDE, "apc.h"))
    return out


def stale() -> bool:
    if not os.path.exists(LIB):
        return True
    t = os.path.getmtime(LIB)
    return any(os.path.getmtime(s) > t for s in sources())


def build(force: bool = False, verbose: bool = False) -> str:
    """Compile libapc.so if missing or older than its sources; return its path."""
    os.makedirs(LIB_DIR, exist_ok=True)
    with open(os.path.join(LIB_DIR, ".lock"), "w") as lk:
        fcntl.flock(lk, fcntl.LOCK_EX)
        if not force and not stale():
            return LIB
        nvcc = os.environ.get("NVCC", "nvcc")
        common = ARCH + ["-O3", "-lineinfo", "-std=c++17", "-Xcompiler", "-fPIC,-fvisibility=hidden",
                         "-I", INCLUDE] + NUMERIC + DEFINES
        if verbose:
            common += ["-Xptxas", "-v"]
        procs, objs = [], []
        for u in UNITS:
            obj = os.path.join(LIB_DIR, u + ".o")
            objs.append(obj)
            procs.append(subprocess.Popen([nvcc, "-c", os.path.join(CSRC, u), "-o", obj] + common,
                                          stdout=subprocess.PIPE, stderr=subprocess.STDOUT, text=True))
        logs = []
        for u, p in zip(UNITS, procs):
            out, _ = p.communicate()
            logs.append(out)
            if p.returncode != 0:
                raise RuntimeError("nvcc failed on %s:\n%s" % (u, out))
        if verbose:
            print("".join(logs))
        tmp = LIB + ".tmp%d" % os.getpid()
        subprocess.run([nvcc] + ARCH + ["-shared", "-o", tmp] + objs, check=True)
        os.replace(tmp, LIB)
    return LIB


def build_probe(force: bool = False) -> str:
    """Compile libapc_probe.so if missing or older than its source; return its path."""
    os.makedirs(BUILD, exist_ok=True)
    with open(os.path.join(BUILD, ".lock_probe"), "w") as lk:
        fcntl.flock(lk, fcntl.LOCK_EX)
        if not force and os.path.exists(PROBE_LIB) and os.path.getmtime(PROBE_LIB) >= os.path.getmtime(PROBE_SRC):
            return PROBE_LIB
        nvcc = os.environ.get("NVCC", "nvcc")
        tmp = PROBE_LIB + ".tmp%d" % os.getpid()
        subprocess.run([nvcc] + ARCH + ["-O3", "-lineinfo", "-std=c++17", "-Xcompiler", "-fPIC,-fvisibility=hidden",
                                        "-shared", PROBE_SRC, "-o", tmp], check=True)
        os.replace(tmp, PROBE_LIB)
    return PROBE_LIB


if __name__ == "__main__":
    import sys
    print(build(force="--force" in sys.argv, verbose="-v" in sys.argv))
