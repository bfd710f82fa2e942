"""Measured integer-pipe rates of the current GPU, from the register-only
probes of ``libapc_probe.so`` (csrc/apc_probe.cu).  The benchmark divides
the verification pass's work, counted from the splitmix64 definition, by
these rates to form its roofline; nothing in the hot path uses them.

``int_rates()`` returns, for each probe kind, the SM's lane-operations per
clock (from the kernel's own clock64 readings, independent of the clock
frequency) and lane-operations per second (from CUDA events on the launching
stream, at whatever clock the GPU ran).
"""
from __future__ import annotations

import ctypes
import statistics

from . import _build

KINDS = {"alu": 0, "fma": 1, "both": 2, "mulhi": 3, "mulwide": 4, "mul64": 5, "mul64x": 6}
OPS_PER_STEP = {"alu": 2, "fma": 2, "both": 4, "mulhi": 2, "mulwide": 2, "mul64": 6, "mul64x": 6}

_lib = None


def library():
    global _lib
    if _lib is None:
        lib = ctypes.CDLL(_build.build_probe())
        lib.apc_probe_int_rate.argtypes = [ctypes.c_int, ctypes.c_uint32, ctypes.c_uint32, ctypes.c_uint32,
                                           ctypes.c_void_p, ctypes.c_void_p]
        lib.apc_probe_int_rate.restype = ctypes.c_int
        lib.apc_probe_threads.restype = ctypes.c_int
        lib.apc_probe_chains.restype = ctypes.c_int
        _lib = lib
    return _lib


def int_rates(iters: int = 8192, reps: int = 5, kinds=("alu", "fma", "both", "mul64", "mul64x")) -> dict:
    """Lane-op rates of the ALU pipe ("alu": funnel shifts and xors), the
    multiply-add pipe ("fma": 32-bit multiply-adds), both together ("both":
    equal numbers, the issue-limited mix) and whole 64-bit multiplies, three
    multiply-add lane-ops each, in the compiler's form ("mul64") and as one
    widening and two plain multiply-adds ("mul64x"), and on request of the
    high ("mulhi") and widening ("mulwide", only the low half used)
    multiply-adds, on a grid of one
    1024-thread CTA per SM; median of ``reps`` launches after one warm-up.
    Per clock: each SM's lane-ops over the span of its SM clock counter from
    its first CTA's start to its last CTA's end, median over the SMs."""
    import torch
    lib = library()
    dev = torch.cuda.current_device()
    sms = torch.cuda.get_device_properties(dev).multi_processor_count
    grid = sms
    threads, chains = lib.apc_probe_threads(), lib.apc_probe_chains()
    clocks = torch.empty(3 * grid + 1, dtype=torch.int64, device="cuda")
    stream = torch.cuda.current_stream()
    out = {"sms": sms, "grid": grid, "threads": threads, "iters": iters}
    for name in kinds:
        kind = KINDS[name]
        per_cta = threads * iters * chains * OPS_PER_STEP[name]
        clk, sec = [], []
        for r in range(reps + 1):
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record(stream)
            rc = lib.apc_probe_int_rate(kind, iters, grid, 0x5EED5EED, ctypes.c_void_p(clocks.data_ptr()),
                                        ctypes.c_void_p(stream.cuda_stream))
            if rc:
                raise RuntimeError("integer-rate probe launch failed (cudaError %d)" % rc)
            e1.record(stream)
            torch.cuda.synchronize()
            if r == 0:
                continue
            c = clocks.cpu().tolist()
            span = {}
            for b in range(grid):
                sm, t0, t1 = c[3 * b], c[3 * b + 1], c[3 * b + 2]
                lo, hi, n = span.get(sm, (t0, t1, 0))
                span[sm] = (min(lo, t0), max(hi, t1), n + 1)
            clk.append(statistics.median(n * per_cta / (hi - lo) for lo, hi, n in span.values()))
            sec.append(grid * per_cta / (e0.elapsed_time(e1) * 1e-3))
        out[name] = {"lane_ops_per_clk_per_sm": statistics.median(clk), "lane_ops_per_s": statistics.median(sec)}
    return out
