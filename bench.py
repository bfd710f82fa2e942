#!/usr/bin/env python3
"""Benchmark of the committed optimizer step with state digest on GB300.

One step = the whole hot path over one rank's shard: ``apc_commit_step``
(fused AdamW + bf16 copy + four digests) followed by the ``apc_digest``
verification pass over the written buffers.  Workload (default): the full
Mistral-7B model on one GPU, 291 separately allocated tensors, 7,248,023,552
elements (~116 GB of fp32 state), optimizer step 18.  The state is larger
than L2 (129 MB), so no flush is needed between timed steps.

Prints one JSON line (rank 0).  ``--impl reference`` times the CPU oracle on
a bounded sample of the same workload instead.

Multi-GPU (torchrun), two partitions (--split):
  copy   (default) rank r commits a full-size copy of the workload's table at
         global offset r * N, so the job's flat model is the concatenation of
         the ranks' copies and per-GPU work is fixed (weak scaling);
  model  rank r commits the contiguous range r of the one model's flat
         parameters (the flat-parameter partition of FSDP), so total work is
         fixed (strong scaling).
There is no collective on the data path.  A Gloo control plane brackets the
timed region with barriers, takes the maximum time over ranks, and after
timing gathers every rank's digests (the whole-model digest is their
wrapping sum) and checks that every verification pass reproduced them.
"""
from __future__ import annotations

import argparse
import hashlib
import json
import os
import statistics
import subprocess
import sys
import threading
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

M64 = (1 << 64) - 1
HP = dict(lr=3e-4, beta1=0.9, beta2=0.95, eps=1e-8, weight_decay=0.1)
METRIC = "commit-step elements/s and HBM GB/s (fraction of GB300 peak), ms per 7.25B-param step"
COMMIT_BYTES = 28   # per element: p, m, v fp32 read+write (24) + bf16 g read (2) + bf16 w write (2)
VERIFY_BYTES = 14   # per element: p, m, v fp32 (12) + bf16 w (2) read
FALLBACK_HBM_GBS = 6800.0


# ----------------------------------------------------------------- helpers

L2_BYTES = 129 << 20          # the GB300's L2
# The verification pass's work per splitmix64 term, counted from the
# definition (first output of SplitMix64 seeded with the key, summed mod
# 2^64) in 32-bit operations:
#   increment            64-bit add                          2 adds
#   z ^= z >> 30, 27, 31 per xor-shift: a funnel shift for the low half, a
#                        shift for the high half, two xors    3 x (1 + 1 + 2)
#   z *= C1, C2          per multiply: low x low widened, the two cross
#                        products into the high word         2 x 3 multiply-adds
#   D += z               64-bit add (one three-input add per half for a pair
#                        of terms)                           1 add
# minus what two identities remove: the high half's first shift is one per
# run of keys whose incremented high words share their top two bits (the
# kernels check this per tile); for a 16-bit word the increment never carries
# and leaves the low half's top bits at 01, so the first funnel shift is the
# single multiply-add 4*hi + 1.  Where the operations can run:
#   xors                       ALU only                           6
#   multiplies                 multiply-add pipe only             6
#   adds, high-word shifts,    either pipe, one op each           5 (fp32 word)
#   and 4*hi + 1                                                  6 (16-bit word)
#   funnel shifts              ALU, or two multiply-adds          3 (fp32), 2 (16-bit)
# 20 operations per term when every flexible one runs on the ALU.
TERM_OPS = {"f32": dict(alu_only=6, mul_only=6, flex=5, funnel=3),
            "bf16": dict(alu_only=6, mul_only=6, flex=6, funnel=2)}
ISSUE_LANES_PER_CLK_PER_SM = 128     # 4 schedulers x one 32-lane warp instruction per clock


def integer_ceiling(words: dict, rates: dict) -> float:
    """Elements per clock per SM at which the integer work of one element
    (``words``: count of fp32 and 16-bit words digested per element) fits
    the measured ALU and multiply-add lane rates and the issue width, with
    the flexible operations split between the two pipes as well as
    possible (a convex piecewise-linear minimum, scanned finely).  The six
    multiply-adds of a term's two 64-bit multiplies run at the measured rate
    of whole 64-bit multiplies, three multiply-adds each, in the faster of
    the two forms probed ("mul64": the compiler's; "mul64x": one widening
    and two plain multiply-adds) when the rates have them, else at the plain
    multiply-add rate."""
    A0 = sum(n * (t["alu_only"] + t["flex"] + t["funnel"]) for k, n in words.items() for t in [TERM_OPS[k]])
    F0 = sum(n * t["mul_only"] for k, n in words.items() for t in [TERM_OPS[k]])
    n1 = sum(n * TERM_OPS[k]["flex"] for k, n in words.items())
    nf = sum(n * TERM_OPS[k]["funnel"] for k, n in words.items())
    ra = rates["alu"]["lane_ops_per_clk_per_sm"]
    rf = rates["fma"]["lane_ops_per_clk_per_sm"]
    m64 = [rates[k]["lane_ops_per_clk_per_sm"] for k in ("mul64", "mul64x") if k in rates]
    rm = max(m64) if m64 else rf
    ri = ISSUE_LANES_PER_CLK_PER_SM
    best = None
    steps = 4000
    for i in range(steps + 1):
        x = (n1 + nf) * i / steps                    # operations moved to the multiply-add pipe
        extra = max(0.0, x - n1)                     # funnel shifts moved cost two multiply-adds each
        t = max((A0 - x) / ra, F0 / rm + (x + extra) / rf, (A0 + F0 + extra) / ri)
        best = t if best is None or t < best else best
    return 1.0 / best


# What each synthetic workload stands for (synth/workloads.py).
WORKLOAD_TEXT = {
    "c1": "one flat shard of 1,048,576 elements",
    "c2": "one Mistral-7B MLP FSDP unit (gate, up, down) as one flat shard",
    "c3": "ragged shard of a 1.216B-parameter decoder for 8 ranks",
    "c4": "Mistral-7B rank shard 9 of 16, crossing tensor boundaries",
    "c5": "full Mistral-7B shard on one GPU",
}


def verify_roofline(rates, clk, n: int, v_ms: float, hbm_peak: float, launches: int, traffic):
    """The verification pass (4 words per element: p', m', v' fp32 and w
    bf16) against the lower of its integer ceiling, from the definition's
    operation count and the measured lane rates at the sampled SM clock, and
    its HBM ceiling (14 bytes per element at the measured copy bandwidth)."""
    terms_per_s = 4 * n / (v_ms * 1e-3)
    rec = {"kernel": "digest_kernel", "achieved": terms_per_s / 1e12, "unit": "T splitmix64 terms/s",
           "launches": launches, "traffic": traffic, "algorithmic_bytes": VERIFY_BYTES * n,
           "hbm_gbs": VERIFY_BYTES * n / (v_ms * 1e-3) / 1e9, "hbm_frac": VERIFY_BYTES * n / (v_ms * 1e-3) / 1e9 / hbm_peak}
    hbm_terms = 4 * hbm_peak * 1e9 / VERIFY_BYTES
    if rates is None:
        rec.update(bound="hbm", peak=hbm_terms / 1e12, frac=terms_per_s / hbm_terms,
                   peak_basis="integer rates not measured: HBM only")
        return rec
    sm_hz = (clk["sm_mhz"] if clk and clk.get("sm_mhz") else 2070.0) * 1e6
    per_clk = integer_ceiling({"f32": 3, "bf16": 1}, rates)            # elements per clock per SM
    int_terms = 4 * per_clk * rates["sms"] * sm_hz
    bound, peak = ("alu", int_terms) if int_terms < hbm_terms else ("hbm", hbm_terms)
    rec.update(bound=bound, peak=peak / 1e12, frac=terms_per_s / peak, integer_peak=int_terms / 1e12,
               integer_frac=terms_per_s / int_terms, hbm_peak_terms=hbm_terms / 1e12,
               measured_lane_ops_per_clk_per_sm={k: rates[k]["lane_ops_per_clk_per_sm"]
                                                 for k in ("alu", "fma", "both", "mul64", "mul64x") if k in rates},
               sm_mhz=sm_hz / 1e6,
               peak_basis="splitmix64 as defined, 20 32-bit operations per term (6 xors on the ALU, the 6 "
                          "multiply-adds of two 64-bit multiplies at the measured rate of whole 64-bit multiplies in their faster form, "
                          "the adds and shifts on either pipe, a funnel shift costing two multiply-adds off the "
                          "ALU), split as well as possible over the ALU and multiply-add lane rates measured by "
                          "register-only probes (libapc_probe.so) and 128 issue lanes per clock per SM, at the "
                          "sampled SM clock; against 14 B/element at the measured HBM bandwidth")
    return rec


def measured_peak():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            return float(json.load(f)["hbm_gbs"]), "measured"
    except (OSError, KeyError, ValueError):
        return FALLBACK_HBM_GBS, "fallback"


# The sources each profiled kernel is compiled from (its translation unit and
# the device headers it includes); host code only launches it.
KERNEL_SOURCES = {
    "commit_kernel": ["apc_commit.cu", "apc_device.cuh", "apc_tma.cuh", "apc_internal.h"],
    "digest_kernel": ["apc_digest.cu", "apc_device.cuh", "apc_internal.h"],
}


def kernel_source_hash(kernel: str) -> str:
    """Hash of a kernel's sources with comments and blank space removed, so
    that its recorded ncu traffic is dropped whenever its code changes."""
    import re
    h = hashlib.sha256()
    csrc = os.path.join(ROOT, "paper_2609_18178_gb300", "csrc")
    for name in KERNEL_SOURCES[kernel]:
        with open(os.path.join(csrc, name)) as f:
            code = f.read()
        code = re.sub(r"/\*.*?\*/", " ", code, flags=re.S)
        code = re.sub(r"//[^\n]*", " ", code)
        code = " ".join(code.split())
        h.update(name.encode() + code.encode())
    return h.hexdigest()[:16]


def profiled_field(kernel: str, field: str):
    """A figure of ``kernel`` from the committed ncu summary, if it was taken
    on the current kernel sources; else None."""
    path = os.path.join(ROOT, "profiles", "traffic.json")
    try:
        with open(path) as f:
            rec = json.load(f)[kernel]
    except (OSError, KeyError, ValueError):
        return None
    src = KERNEL_SOURCES.get(kernel.replace("_bf16", ""))
    if src is None or rec.get("source_hash") != kernel_source_hash(kernel.replace("_bf16", "")):
        return None
    return rec.get(field)


def issue_ceiling(kernel: str, n: int, ms: float, sms: int, clk) -> dict | None:
    """The instruction-issue ceiling of a commit launch: its ncu instruction
    count per element x elements over 128 issue lanes per clock per SM at the
    sampled SM clock."""
    ipe = profiled_field(kernel, "inst_per_element")
    if ipe is None:
        return None
    sm_hz = (clk["sm_mhz"] if clk and clk.get("sm_mhz") else 2070.0) * 1e6
    t = ipe * n / (sms * ISSUE_LANES_PER_CLK_PER_SM * sm_hz)
    return {"inst_per_element": ipe, "ceiling_ms": t * 1e3, "frac": t * 1e3 / ms, "sm_mhz": sm_hz / 1e6}


def profiled_traffic(kernel: str, workload: str):
    """DRAM bytes of one launch (the commit) or one pass (the verification,
    whatever its launch count) of ``kernel`` from the committed ncu summary,
    if it was taken on the current kernel sources; else None."""
    path = os.path.join(ROOT, "profiles", "traffic.json")
    try:
        with open(path) as f:
            rec = json.load(f)[kernel]
    except (OSError, KeyError, ValueError):
        return None
    if rec.get("source_hash") != kernel_source_hash(kernel):
        return None
    if rec.get("workload") != workload:
        return None
    return rec.get("dram_bytes_per_launch", rec.get("dram_bytes_per_pass"))


class ClockSampler:
    """nvidia-smi clock/throttle samples during the timed region."""
    FIELDS = ["clocks.sm", "clocks.max.sm", "clocks_event_reasons.hw_slowdown",
              "clocks_event_reasons.hw_thermal_slowdown", "clocks_event_reasons.sw_thermal_slowdown",
              "clocks_event_reasons.sw_power_cap", "power.draw"]

    def __init__(self, device_index: int):
        self.proc = None
        self.lines = []
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(device_index), "--query-gpu=" + ",".join(self.FIELDS),
                 "--format=csv,noheader,nounits", "-lms", "100"],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            self.thread = threading.Thread(target=self._read, daemon=True)
            self.thread.start()
        except OSError:
            self.proc = None

    def _read(self):
        for line in self.proc.stdout:
            self.lines.append(line.strip())

    def stop(self):
        if self.proc is None:
            return None
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        self.thread.join(timeout=5)
        sm, smax, reasons, power = [], None, set(), []
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for line in self.lines:
            parts = [x.strip() for x in line.split(",")]
            if len(parts) != len(self.FIELDS):
                continue
            try:
                sm.append(float(parts[0]))
                smax = float(parts[1])
                power.append(float(parts[6]))
            except ValueError:
                continue
            for nm, val in zip(names, parts[2:6]):
                if val.lower() == "active":
                    reasons.add(nm)
        if not sm:
            return None
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": smax, "reasons": sorted(reasons),
                "samples": len(sm), "power_w_max": max(power) if power else None}


# -------------------------------------------------------- distributed setup

def dist_env():
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return world, rank, local


def init_control_plane(world: int):
    """Gloo process group for barriers and the post-step digest exchange."""
    if world <= 1:
        return None
    import torch.distributed as dist
    dist.init_process_group("gloo")
    return dist


def barrier(dist):
    if dist is not None:
        dist.barrier()


def max_over_ranks(dist, x: float) -> float:
    if dist is None:
        return x
    import torch
    t = torch.tensor([x], dtype=torch.float64)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def shard_offset(rank: int, elements_per_rank: int) -> int:
    """Global index of rank r's first element: the job's flat model is the
    concatenation of the ranks' equally sized shards (weak scaling)."""
    return rank * elements_per_rank


def exchange_digests(dist, step: int, commit_digests: list[int], verify_digests: list[int], shard: int):
    """Post-step control-plane exchange: every rank reports (frontier =
    optimizer step, generation 0, its 4 commit digests, whether its
    verification pass reproduced them) and the cohort checks agreement
    (paper_2609_18178_gb300.cohort).  Returns (whole-model digests = wrapping
    sum over the shards, all verified); raises cohort.CohortError otherwise."""
    commit = [int(d) & M64 for d in commit_digests]
    ok = commit == [int(d) & M64 for d in verify_digests]
    if dist is None:
        return commit, ok
    from paper_2609_18178_gb300 import cohort
    ag = cohort.agree(dist, frontier=step, generation=0, digests=commit, shard=shard, verified=ok)
    return ag.whole_digests, True


def sum_over_ranks(dist, digests: list[int]) -> list[int]:
    """Digests added over the ranks mod 2^64 (the whole model's, by
    concatenation): a control-plane all-reduce of int64 bit patterns, whose
    sum wraps exactly as the unsigned sum does."""
    d = [int(x) & M64 for x in digests]
    if dist is None:
        return d
    import torch
    t = torch.tensor([x - (1 << 64) if x >= 1 << 63 else x for x in d], dtype=torch.int64)
    dist.all_reduce(t, op=dist.ReduceOp.SUM)
    return [int(x) & M64 for x in t.tolist()]


def group_pieces(sizes: list[int], n_groups: int) -> list[list[int]]:
    """Consecutive runs of table entries with about equal element counts."""
    total = sum(sizes)
    groups, cur, acc = [], [], 0
    for k, n in enumerate(sizes):
        cur.append(k)
        acc += n
        if acc >= total * (len(groups) + 1) / n_groups and len(groups) < n_groups - 1:
            groups.append(cur)
            cur = []
    if cur:
        groups.append(cur)
    return groups


# ----------------------------------------------- replica verification (f4)

def _replica_main(idx: int, n_rep: int, port: int, workload: str, flip: int, q) -> None:
    """One replica of a hybrid-sharding replication group on the current
    GPU: commit its (identical) shard, then verify and agree with the other
    replicas twice; before the second agreement one bit of replica `flip`'s
    HBM state is flipped through a host-side copy.  Spawned, so it builds its own
    CUDA context; replicas never wait on each other's kernels, only on the
    host control plane."""
    import datetime
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    try:
        import torch
        import torch.distributed as dist
        import paper_2609_18178_gb300 as apc
        from paper_2609_18178_gb300 import cohort
        import synth
        from synth import workloads as W
        dist.init_process_group("gloo", rank=idx, world_size=n_rep, timeout=datetime.timedelta(seconds=300))
        grp = dist.new_group(ranks=list(range(n_rep)), backend="gloo", timeout=datetime.timedelta(seconds=60))
        torch.cuda.set_device(0)
        w = W.ALL[workload]()
        step = w.steps[-1]
        s = torch.cuda.current_stream().cuda_stream
        bufs, goff = [], {}
        for pc in w.pieces:
            goff.setdefault(pc.alloc, pc.goff - pc.at)
        for a, n in enumerate(w.allocs):
            b = {k: torch.empty(n, dtype=torch.float32 if k in "pmv" else torch.int16, device="cuda")
                 for k in "pmvgw"}
            for k, kind in (("p", synth.P), ("m", synth.M), ("v", synth.V)):
                synth.fill_dev(kind, b[k].data_ptr(), n, goff[a], stream=s)
            synth.fill_dev(synth.G, b["g"].data_ptr(), n, goff[a], step=step, stream=s)
            bufs.append(b)
        entries, vbufs = [], []
        for pc in w.pieces:
            b = bufs[pc.alloc]
            sl = slice(pc.at, pc.at + pc.n)
            entries.append(apc.TensorEntry(b["p"][sl], b["m"][sl], b["v"][sl], b["g"][sl], b["w"][sl], pc.goff))
            vbufs += apc.state_buffers(b["p"][sl], b["m"][sl], b["v"][sl], b["w"][sl], pc.goff)
        dc = apc.digests_to_host(apc.commit_step(entries, step, HP))
        passes = []
        for r, flip_here in enumerate((False, idx == flip)):
            if flip_here:
                word = bufs[0]["p"][12345:12346].view(torch.int32).cpu()
                word ^= 1 << 7
                bufs[0]["p"][12345:12346].view(torch.int32).copy_(word)    # host-side fault injection
            dist.barrier(group=grp)
            torch.cuda.synchronize()
            t0 = time.perf_counter()
            dv = apc.digests_to_host(apc.digest(vbufs, 4))
            t1 = time.perf_counter()
            try:
                ag = cohort.agree(dist, step, 1, dv, shard=0, group=grp)
                passes.append(("agreed", ["%016x" % d for d in ag.whole_digests], (t1 - t0) * 1e3,
                               ag.seconds * 1e3))
            except cohort.CohortMismatch as e:
                passes.append(("mismatch", (e.what, e.ranks), (t1 - t0) * 1e3, (time.perf_counter() - t1) * 1e3))
        q.put((idx, dc, passes))
        dist.destroy_process_group()
    except Exception as e:  # reported, never hangs the parent
        q.put((idx, None, "error: %r" % (e,)))


def replica_check(n_rep: int = 4, workload: str = "c4", flip: int = 3, timeout_s: float = 600.0) -> dict:
    """Run the replica verification with n_rep spawned processes on GPU 0."""
    import multiprocessing as mp
    import socket
    with socket.socket() as sk:
        sk.bind(("127.0.0.1", 0))
        port = sk.getsockname()[1]
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    ps = [ctx.Process(target=_replica_main, args=(i, n_rep, port, workload, flip, q)) for i in range(n_rep)]
    t0 = time.perf_counter()
    for p in ps:
        p.start()
    res = []
    try:
        for _ in ps:
            res.append(q.get(timeout=timeout_s))
    finally:
        for p in ps:
            p.join(timeout=60)
            if p.is_alive():
                p.kill()
    res.sort(key=lambda x: x[0])
    errors = [r[2] for r in res if isinstance(r[2], str)]
    if errors:
        return {"replicas": n_rep, "error": errors[0]}
    commit_equal = all(r[1] == res[0][1] for r in res)
    clean_pass = [r[2][0] for r in res]
    flip_pass = [r[2][1] for r in res]
    return {"replicas": n_rep, "workload": workload, "commit_digests_equal": commit_equal,
            "clean_agreed": all(o[0] == "agreed" for o in clean_pass),
            "flipped_replica": flip,
            "flip_detected_by_all": all(o[0] == "mismatch" for o in flip_pass),
            "flip_diagnosis": flip_pass[0][1] if flip_pass[0][0] == "mismatch" else None,
            "verify_ms_max": max(o[2] for o in clean_pass), "agree_ms_max": max(o[3] for o in clean_pass),
            "wall_s": time.perf_counter() - t0}


# ------------------------------------------------------------- GPU arm

def run_gpu(args):
    import torch
    import paper_2609_18178_gb300 as apc
    import synth
    from synth import workloads as W

    world, rank, local = dist_env()
    dist = init_control_plane(world)
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    whole = W.ALL[args.workload]()
    step_t = whole.steps[-1]
    if args.split == "model":
        # flat-parameter partition: rank r commits the contiguous range r of
        # the one model (total work fixed as ranks are added)
        w = W.shard(whole, rank, world)
        base, N_job = 0, whole.n
    else:
        # every rank commits a full-size copy at global offset r * N: the
        # job's flat model is the concatenation of the copies
        w = whole
        base, N_job = shard_offset(rank, whole.n), world * whole.n
    N = w.n

    # resident state: one allocation per tensor, filled by the device generator
    stream = torch.cuda.current_stream()
    s = stream.cuda_stream
    bufs = []
    goff_of = {}
    for pc in w.pieces:
        goff_of.setdefault(pc.alloc, base + pc.goff - pc.at)
    for a, n in enumerate(w.allocs):
        b = dict(p=torch.empty(n, dtype=torch.float32, device=dev), m=torch.empty(n, dtype=torch.float32, device=dev),
                 v=torch.empty(n, dtype=torch.float32, device=dev), g=torch.empty(n, dtype=torch.int16, device=dev),
                 w=torch.empty(n, dtype=torch.int16, device=dev))
        g0 = goff_of[a]
        synth.fill_dev(synth.P, b["p"].data_ptr(), n, g0, stream=s)
        synth.fill_dev(synth.M, b["m"].data_ptr(), n, g0, stream=s)
        synth.fill_dev(synth.V, b["v"].data_ptr(), n, g0, stream=s)
        synth.fill_dev(synth.G, b["g"].data_ptr(), n, g0, step=step_t, stream=s)
        bufs.append(b)
    entries, vbufs = [], []
    for pc in w.pieces:
        b = bufs[pc.alloc]
        sl = slice(pc.at, pc.at + pc.n)
        entries.append(apc.TensorEntry(b["p"][sl], b["m"][sl], b["v"][sl], b["g"][sl], b["w"][sl], base + pc.goff))
        vbufs += apc.state_buffers(b["p"][sl], b["m"][sl], b["v"][sl], b["w"][sl], base + pc.goff)
    out_c = torch.empty(4, dtype=torch.int64, device=dev)
    out_v = torch.empty(4, dtype=torch.int64, device=dev)
    # the table and the buffer list are marshalled once, as a training job
    # would: no Python work sits between a timed event and its launch
    tab, vtab = apc.prepare_table(entries), apc.prepare_buffers(vbufs)
    torch.cuda.synchronize()
    # The first commit runs from the generated state, the same step the
    # oracle computes from the same generated inputs in cpu_baseline's c5
    # stream; later steps update the state in place.
    first_digests = apc.digests_to_host(apc.commit_step(tab, step_t, HP, stream=s, out=out_c))

    user_limit = os.environ.get("APC_GRID_LIMIT")

    def grid_limit(n):
        # APC_GRID_LIMIT is read by every library call (include/apc.h); 0
        # restores whatever the caller of the bench had set
        if n:
            os.environ["APC_GRID_LIMIT"] = str(n)
        elif user_limit is None:
            os.environ.pop("APC_GRID_LIMIT", None)
        else:
            os.environ["APC_GRID_LIMIT"] = user_limit

    def one_step(ev=None):
        if ev is not None:
            ev[0].record(stream)
        apc.commit_step(tab, step_t, HP, stream=s, out=out_c)
        if ev is not None:
            ev[1].record(stream)
        apc.digest(vtab, 4, stream=s, out=out_v)
        if ev is not None:
            ev[2].record(stream)

    if args.schedule == "pipelined":
        # The table cut into groups; the verification of group g runs on a
        # second stream once group g's commit is done, beside the commits of
        # the later groups.  ev[1] marks the end of the last commit, ev[2] the
        # end of the last verification.
        pgroups = group_pieces([pc.n for pc in w.pieces], args.groups)
        ptab = [apc.prepare_table([entries[k] for k in idx]) for idx in pgroups]
        pvtab = [apc.prepare_buffers([vbufs[4 * k + j] for k in idx for j in range(4)]) for idx in pgroups]
        pout = torch.empty(len(pgroups), 8, dtype=torch.int64, device=dev)
        vstream = torch.cuda.Stream(device=dev)
        pdone = [torch.cuda.Event() for _ in pgroups]

        def one_step(ev=None):  # noqa: F811 (the pipelined schedule replaces the sequential one)
            if ev is not None:
                ev[0].record(stream)
            for gi in range(len(pgroups)):
                grid_limit(args.commit_grid)
                apc.commit_step(ptab[gi], step_t, HP, stream=s, out=pout[gi, :4])
                pdone[gi].record(stream)
                vstream.wait_event(pdone[gi])
                grid_limit(args.verify_grid)
                apc.digest(pvtab[gi], 4, stream=vstream.cuda_stream, out=pout[gi, 4:])
            grid_limit(0)
            if ev is not None:
                ev[1].record(stream)
            stream.wait_stream(vstream)
            out_c.copy_(pout[:, :4].sum(0))
            out_v.copy_(pout[:, 4:].sum(0))
            if ev is not None:
                ev[2].record(stream)

    for _ in range(args.warmup):
        one_step()
    torch.cuda.synchronize()

    K = args.steps
    evs = [[torch.cuda.Event(enable_timing=True) for _ in range(3)] for _ in range(K)]
    # A step whose bytes fit in L2 would find its inputs there: write a
    # buffer twice the L2's size between timed steps, outside their events.
    flush = (torch.empty(2 * L2_BYTES // 4, dtype=torch.int32, device=dev)
             if (COMMIT_BYTES + VERIFY_BYTES) * N <= 4 * L2_BYTES else None)
    clocks = ClockSampler(local) if not args.no_clocks else None
    barrier(dist)
    torch.cuda.synchronize()
    for k in range(K):
        if flush is not None:
            flush.fill_(k)
        one_step(evs[k])
    torch.cuda.synchronize()
    barrier(dist)
    clk = clocks.stop() if clocks else None
    rates = None
    if rank == 0:
        try:
            from paper_2609_18178_gb300 import peak as apc_peak
            rates = apc_peak.int_rates()
        except (OSError, RuntimeError, subprocess.CalledProcessError) as ex:
            print("note: integer-rate probe unavailable (%s); verify roofline against HBM only" % ex, file=sys.stderr)
    commit_ms = [evs[k][0].elapsed_time(evs[k][1]) for k in range(K)]
    verify_ms = [evs[k][1].elapsed_time(evs[k][2]) for k in range(K)]
    if flush is None:
        total_ms = evs[0][0].elapsed_time(evs[K - 1][2])
    else:   # per-step events only: the flushes between them are not timed
        total_ms = sum(evs[k][0].elapsed_time(evs[k][2]) for k in range(K))
    total_ms = max_over_ranks(dist, total_ms)
    ms_per_step = total_ms / K
    digests_c = apc.digests_to_host(out_c)
    digests_v = apc.digests_to_host(out_v)
    whole_d, verified = exchange_digests(dist, step_t, digests_c, digests_v, shard=rank)
    first_whole = sum_over_ranks(dist, first_digests)

    # End to end: every step brings its gradient from pinned host memory and
    # returns the digests.  The table is cut into groups of about equal size;
    # a copy stream moves group g's gradient while the compute stream commits
    # and verifies earlier groups (events order each group's kernels after its
    # upload, and each upload after the previous step's commit of that group
    # has read the old gradient), and the host adds the per-group digests
    # (concatenation).  By default the upload is apc_upload: a few CTAs load
    # the pinned host gradient over the host link, on SMs that the step's
    # kernels leave free (apc_set_reserved_sms); --e2e-upload copy uses the
    # DMA copy engines (cudaMemcpyAsync per tensor) instead.
    e2e = None
    host_g = []
    if not args.no_e2e:
        # every rank pins its own copy of the gradient; the leg runs only if
        # all ranks could (a rank without it would leave the others waiting)
        why = ""
        try:
            for b in bufs:
                hg = torch.empty(b["g"].numel(), dtype=torch.int16, pin_memory=True)
                hg.copy_(b["g"])
                host_g.append(hg)
        except RuntimeError as ex:
            host_g, why = [], (str(ex).splitlines() or [type(ex).__name__])[0]
        if max_over_ranks(dist, 0.0 if why == "" else 1.0) > 0:
            e2e = {"error": "pinned host memory for the gradient (%.1f GB per rank) could not be allocated on "
                            "every rank%s" % (2 * N / 1e9, ": " + why if why else "")}
    if not args.no_e2e and e2e is None:
        groups = group_pieces([pc.n for pc in w.pieces], args.e2e_groups)
        n_groups = len(groups)
        copy_stream = torch.cuda.Stream(device=dev)
        outs = torch.empty(n_groups, 8, dtype=torch.int64, device=dev)
        host_out = torch.empty(n_groups, 8, dtype=torch.int64, pin_memory=True)
        ready = [torch.cuda.Event() for _ in range(n_groups)]
        done = [torch.cuda.Event() for _ in range(n_groups)]
        gtab = [apc.prepare_table([entries[k] for k in idx]) for idx in groups]
        gvtab = [apc.prepare_buffers([vbufs[4 * k + j] for k in idx for j in range(4)]) for idx in groups]

        def segments(idx):
            return [apc.Segment(bufs[w.pieces[k].alloc]["g"][w.pieces[k].at:w.pieces[k].at + w.pieces[k].n],
                                host_g[w.pieces[k].alloc][w.pieces[k].at:w.pieces[k].at + w.pieces[k].n])
                    for k in idx]

        gseg = [apc.prepare_segments(segments(idx)) for idx in groups]
        use_sm = args.e2e_upload == "sm"

        def upload(gi, idx):
            if use_sm:
                apc.upload(gseg[gi], args.e2e_upload_ctas, stream=copy_stream)
                return
            with torch.cuda.stream(copy_stream):
                for k in idx:
                    pc = w.pieces[k]
                    bufs[pc.alloc]["g"][pc.at:pc.at + pc.n].copy_(host_g[pc.alloc][pc.at:pc.at + pc.n],
                                                                  non_blocking=True)

        def e2e_step():
            # group g's upload for this step waits only until the previous
            # step's commit of group g has read its gradient (done[g])
            for gi, idx in enumerate(groups):
                copy_stream.wait_event(done[gi])
                upload(gi, idx)
                ready[gi].record(copy_stream)
                stream.wait_event(ready[gi])
                apc.commit_step(gtab[gi], step_t, HP, stream=s, out=outs[gi, :4])
                done[gi].record(stream)
                apc.digest(gvtab[gi], 4, stream=s, out=outs[gi, 4:])
            host_out.copy_(outs, non_blocking=True)

        if use_sm:
            apc.set_reserved_sms(args.e2e_reserved_sms)
        torch.cuda.synchronize()
        for _ in range(max(1, args.warmup)):
            e2e_step()
        torch.cuda.synchronize()
        ke = max(1, args.e2e_steps)
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        barrier(dist)
        torch.cuda.synchronize()
        step_ev = [torch.cuda.Event(enable_timing=True) for _ in range(ke)]
        e0.record(stream)
        copy_stream.wait_event(e0)
        for k in range(ke):
            e2e_step()
            step_ev[k].record(stream)
        e1.record(stream)
        torch.cuda.synchronize()
        barrier(dist)
        apc.set_reserved_sms(0)
        e2e_ms = max_over_ranks(dist, e0.elapsed_time(e1)) / ke
        step_ms = [e0.elapsed_time(step_ev[0])] + [step_ev[k - 1].elapsed_time(step_ev[k]) for k in range(1, ke)]
        got = [[int(x) & M64 for x in row] for row in host_out.tolist()]
        e2e_verified = all(r[:4] == r[4:] for r in got)

        def upload_alone(sm):
            # the whole gradient with nothing else running: the bound of the end-to-end step
            h0, h1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            h0.record(copy_stream)
            if sm:
                apc.upload(apc.prepare_segments(segments(range(len(w.pieces)))), args.e2e_upload_ctas,
                           stream=copy_stream)
            else:
                with torch.cuda.stream(copy_stream):
                    for pc in w.pieces:
                        bufs[pc.alloc]["g"][pc.at:pc.at + pc.n].copy_(host_g[pc.alloc][pc.at:pc.at + pc.n],
                                                                      non_blocking=True)
            h1.record(copy_stream)
            torch.cuda.synchronize()
            return h0.elapsed_time(h1)

        h2d_ms = upload_alone(use_sm)
        ce_ms = upload_alone(False) if use_sm else h2d_ms
        e2e = {"value": N_job / (e2e_ms * 1e-3), "unit": "elements/s",
               "h2d_bytes_per_step": 2 * N, "d2h_bytes_per_step": 64 * n_groups, "ms_per_step": e2e_ms,
               "steps": ke, "groups": n_groups, "verify_matches_commit": e2e_verified,
               "upload": ({"method": "apc_upload: SM loads of pinned host memory over the host link",
                           "ctas": args.e2e_upload_ctas, "reserved_sms": args.e2e_reserved_sms} if use_sm else
                          {"method": "cudaMemcpyAsync per tensor (DMA copy engines)"}),
               "h2d_alone_ms": h2d_ms, "h2d_alone_gbs": 2 * N / (h2d_ms * 1e-3) / 1e9,
               "copy_engine_alone_ms": ce_ms,
               "step_ms": [round(x, 2) for x in step_ms], "median_step_ms": statistics.median(step_ms),
               "note": "copy-engine transfers on this machine stall for tens to hundreds of ms about twice a "
                       "second; SM loads over the host link do not"}
        del host_g

    # Next rows measured beside the step: the fused commit that also zeroes
    # the gradients (30 B/element) and the quiescence guard over the
    # gradients (2 B/element).  Run last: they leave the gradients zeroed.
    nxt = None
    if not args.no_next:
        gbufs = apc.prepare_buffers([apc.BufferEntry(bufs[pc.alloc]["g"][pc.at:pc.at + pc.n], 0, 0, apc.BF16)
                                     for pc in w.pieces])
        out_n = torch.empty(1, dtype=torch.int64, device=dev)

        def timed(fn, reps):
            for _ in range(2):
                fn()
            torch.cuda.synchronize()
            ms = []
            for _ in range(reps):
                a0, a1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
                a0.record(stream)
                fn()
                a1.record(stream)
                torch.cuda.synchronize()
                ms.append(a0.elapsed_time(a1))
            return statistics.median(ms)

        sms = torch.cuda.get_device_properties(dev).multi_processor_count
        sm_hz = (clk["sm_mhz"] if clk and clk.get("sm_mhz") else 2070.0) * 1e6
        nz_before = apc.digests_to_host(apc.count_nonzero(gbufs, 1, stream=s, out=out_n))[0]
        guard_ms = timed(lambda: apc.count_nonzero(gbufs, 1, stream=s, out=out_n), max(3, K))
        zero_ms = timed(lambda: apc.commit_step(tab, step_t, HP, stream=s, out=out_c, zero_grad=True), max(3, K))
        nz_after = apc.digests_to_host(apc.count_nonzero(gbufs, 1, stream=s, out=out_n))[0]
        peak_n, _ = measured_peak()
        torch.cuda.synchronize()
        # f3: the paper's bf16-state rank shard (rank 1 of 4), committed and verified
        w3 = W.f3()
        if args.f3_tensors:    # the first K tensors only (a smaller case for profiling)
            kept = w3.pieces[:args.f3_tensors]
            w3 = W.Workload(w3.name, kept, w3.steps, w3.chained, w3.verify, [max(pc.at + pc.n for pc in kept)])
        N3 = w3.n
        b3 = {k: torch.empty(N3, dtype=torch.int16, device=dev) for k in "pmvg"}
        g3 = w3.pieces[0].goff - w3.pieces[0].at
        for k, kind in (("p", synth.P16), ("m", synth.M16), ("v", synth.V16)):
            synth.fill_dev(kind, b3[k].data_ptr(), N3, g3, stream=s)
        synth.fill_dev(synth.G, b3["g"].data_ptr(), N3, g3, step=w3.steps[0], stream=s)
        e3, v3 = [], []
        for pc in w3.pieces:
            sl = slice(pc.at, pc.at + pc.n)
            e3.append(apc.TensorEntryBF16(b3["p"][sl], b3["m"][sl], b3["v"][sl], b3["g"][sl], pc.goff))
            v3 += apc.state_buffers_bf16(b3["p"][sl], b3["m"][sl], b3["v"][sl], pc.goff)
        e3, v3 = apc.prepare_table(e3), apc.prepare_buffers(v3)
        out3 = torch.empty(3, dtype=torch.int64, device=dev)
        out3v = torch.empty(3, dtype=torch.int64, device=dev)
        f3_ms = timed(lambda: apc.commit_step_bf16(e3, w3.steps[0], HP, stream=s, out=out3), max(3, K))
        f3v_ms = timed(lambda: apc.digest(v3, 3, stream=s, out=out3v), max(3, K))
        f3_ok = apc.digests_to_host(out3) == apc.digests_to_host(out3v)
        del b3, e3, v3
        nxt = {"f3_commit_bf16_state": {"workload": "rank 1 of 4 of Mistral-7B, %d elements, %d pieces, bf16 p/m/v"
                                                    % (N3, len(w3.pieces)), "ms": f3_ms, "gbs": 14 * N3 / (f3_ms * 1e-3) / 1e9,
                                        "frac": 14 * N3 / (f3_ms * 1e-3) / 1e9 / peak_n, "bytes_per_element": 14,
                                        "verify_ms": f3v_ms, "verify_gbs": 6 * N3 / (f3v_ms * 1e-3) / 1e9,
                                        "verify_frac": 6 * N3 / (f3v_ms * 1e-3) / 1e9 / peak_n,
                                        "verify_matches_commit": f3_ok,
                                        "issue": issue_ceiling("commit_kernel_bf16", N3, f3_ms, sms, clk),
                                        "verify_integer": (None if rates is None else
                                                           {"ceiling_ms": 1e3 * N3 / (integer_ceiling({"bf16": 3}, rates)
                                                                                     * rates["sms"] * sm_hz),
                                                            "frac": 1e3 * N3 / (integer_ceiling({"bf16": 3}, rates)
                                                                                * rates["sms"] * sm_hz) / f3v_ms})},
               "f1_commit_zero_grad": {"ms": zero_ms, "gbs": 30 * N / (zero_ms * 1e-3) / 1e9,
                                       "frac": 30 * N / (zero_ms * 1e-3) / 1e9 / peak_n, "bytes_per_element": 30},
               "f1_guard_count_nonzero": {"ms": guard_ms, "gbs": 2 * N / (guard_ms * 1e-3) / 1e9,
                                          "frac": 2 * N / (guard_ms * 1e-3) / 1e9 / peak_n, "bytes_per_element": 2,
                                          "nonzero_before": nz_before, "nonzero_after_zeroing": nz_after}}

    cpu, oracle_c5 = None, None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        cpu, oracle_c5 = cpu_baseline(os.cpu_count() or 1, plan_c5=args.cpu_plan == "full")

    if rank == 0 and world == 1 and not args.no_next and args.replicas > 1:
        # the c5 state stays resident (116 GB); the replicas add 4 x 7.3 GB
        torch.cuda.synchronize()
        torch.cuda.empty_cache()
        f4 = replica_check(args.replicas, "c4", flip=args.replicas - 1)
        if nxt is not None:
            nxt["f4_replica_verify"] = f4

    if rank != 0:
        if dist is not None:
            dist.destroy_process_group()
        return
    peak, peak_kind = measured_peak()
    n_commit_launches = max(1, (len(entries) + 439) // 440)
    n_digest_launches = max(1, (len(vbufs) + 999) // 1000)
    if args.schedule == "pipelined":
        n_commit_launches = n_digest_launches = len(group_pieces([pc.n for pc in w.pieces], args.groups))
    c_ms = statistics.median(commit_ms)
    v_ms = statistics.median(verify_ms)
    c_avg = sum(commit_ms) / K
    v_avg = sum(verify_ms) / K
    achieved = COMMIT_BYTES * N / (c_avg * 1e-3) / 1e9
    line = {
        "metric": METRIC,
        "value": N_job / (ms_per_step * 1e-3),
        "unit": "elements/s",
        "n_gpus": world,
        "steps": K,
        "warmup": args.warmup,
        "ms_per_step": ms_per_step,
        "higher_is_better": True,
        "scaling": "strong" if args.split == "model" else "weak",
        "vs_baseline": None,
        "dtype": "f32+u64",
        "data": "synthetic",
        "config": {"workload": "%s: %s, %d tensors, %d elements, step %d, commit+digest then re-verify"
                               % (whole.name, WORKLOAD_TEXT.get(whole.name, "synthetic shard"), len(whole.pieces),
                                  whole.n, step_t),
                   "elements": N_job, "elements_per_rank": N, "tensors": len(whole.pieces), "step": step_t,
                   "split": args.split,
                   "parallelism": ("%d ranks x one contiguous range of the flat model each (no data-path "
                                   "collective)" % world if args.split == "model" else
                                   "%d ranks x one full-size shard each (no data-path collective)" % world),
                   "l2": ("inputs larger than L2 (%.1f GB resident state)" % (16 * N / 1e9) if flush is None else
                          "L2 flushed between timed steps (a %d MB write outside the step's events): the step's "
                          "%.3f GB would otherwise fit in L2" % (2 * L2_BYTES >> 20,
                                                                  (COMMIT_BYTES + VERIFY_BYTES) * N / 1e9))},
        "hbm_gbs_step": (COMMIT_BYTES + VERIFY_BYTES) * N / (ms_per_step * 1e-3) / 1e9,
        "commit_ms": c_ms,
        "verify_ms": v_ms,
        "commit_gbs": COMMIT_BYTES * N / (c_ms * 1e-3) / 1e9,
        "verify_gbs": VERIFY_BYTES * N / (v_ms * 1e-3) / 1e9,
        "commit_elements_per_s": N / (c_ms * 1e-3),
        "frac_of_spec_8tbs": achieved / 8000.0,
        "roofline": None if args.schedule == "pipelined" else {"bound": "hbm", "kernel": "commit_kernel",
                     "achieved": achieved, "peak": peak,
                     "peak_kind": peak_kind, "unit": "GB/s", "frac": achieved / peak,
                     "frac_of_spec_8tbs": achieved / 8000.0,
                     "traffic": profiled_traffic("commit_kernel", w.name),
                     "traffic_note": ("ncu DRAM bytes of the 152M-element c3 launch scaled by elements: a lower "
                                      "bound, since writes still in L2 when that launch ended are not counted"),
                     "algorithmic_bytes_per_launch": COMMIT_BYTES * N,
                     "issue": issue_ceiling("commit_kernel", N, c_avg, torch.cuda.get_device_properties(dev)
                                            .multi_processor_count, clk)},
        "roofline_verify": None if args.schedule == "pipelined" else verify_roofline(
            rates, clk, N, v_avg, peak, n_digest_launches, profiled_traffic("digest_kernel", w.name)),
        "schedule": ({"kind": "sequential"} if args.schedule == "sequential" else
                     {"kind": "pipelined", "groups": args.groups, "commit_grid": args.commit_grid or "default",
                      "verify_grid": args.verify_grid or "default", "commit_span_ms": c_ms,
                      "verify_tail_ms": v_ms,
                      "note": "commit and verification kernels overlap: commit_ms is the span of the commit "
                              "stream, verify_ms the verification tail after it, and the kernel rooflines are "
                              "those of the sequential schedule, not measured here"}),
        "gpu_launches": K * (n_commit_launches + n_digest_launches),
        "gpu_launches_note": "per timed step: %d commit_kernel + %d digest_kernel launches (%d tensors, %d buffers; "
                             "up to 440 tensors and 1000 buffers per launch)"
                             % (n_commit_launches, n_digest_launches, len(entries), len(vbufs)),
        "digests": ["%016x" % d for d in whole_d],
        "first_commit_digests": ["%016x" % d for d in first_whole],
        "oracle_parity": (None if oracle_c5 is None or whole.name != "c5" or world != 1 else
                          {"workload": "c5", "step": step_t,
                           "gpu_first_commit_digests": ["%016x" % d for d in first_digests],
                           "oracle_digests": ["%016x" % d for d in oracle_c5],
                           "equal": first_digests == oracle_c5,
                           "what": "digests of p', m', v', w after one step from the generated state: the GPU's "
                                   "first (untimed) commit against the oracle streamed over every element"}),
        "verify_matches_commit": verified,
        "clocks": clk,
        "e2e": e2e,
        "cpu_baseline": cpu,
        "next_rows": nxt,
    }
    print(json.dumps(line), flush=True)
    if dist is not None:
        dist.destroy_process_group()


# --------------------------------------------------------- CPU oracle arm

def cpu_model() -> str:
    """The host CPU's model name (lscpu, else /proc/cpuinfo, else the architecture)."""
    try:
        out = subprocess.run(["lscpu"], capture_output=True, text=True, timeout=10).stdout
        for line in out.splitlines():
            if line.strip().startswith("Model name:"):
                return line.split(":", 1)[1].strip()
    except (OSError, subprocess.SubprocessError):
        pass
    try:
        with open("/proc/cpuinfo") as f:
            for line in f:
                if line.lower().startswith("model name"):
                    return line.split(":", 1)[1].strip()
    except OSError:
        pass
    import platform
    return platform.machine()


def _oracle_step(p, m, v, g, g0: int, h8, threads: int, pool=None):
    """One oracle step over the contiguous global range [g0, g0 + n): the
    committed step (the oracle's own threaded partition when threads > 1),
    then the verification digests of the four written buffers (chunks on
    ``pool`` when threads > 1).  Updates p, m, v in place.  Returns
    (commit seconds, verify seconds, commit digests, verification matches)."""
    import oracle
    n = p.size
    t0 = time.perf_counter()
    wb, d = oracle.commit(p, m, v, g, g0, h8, nthreads=threads)
    t1 = time.perf_counter()
    if threads <= 1 or pool is None:
        dv = [oracle.digest_f32(p, g0), oracle.digest_f32(m, g0), oracle.digest_f32(v, g0), oracle.digest_u16(wb, g0)]
    else:
        chunk = -(-n // threads)
        parts = []
        for lo in range(0, n, chunk):
            hi = min(n, lo + chunk)
            parts += [(oracle.digest_f32, p[lo:hi], lo), (oracle.digest_f32, m[lo:hi], lo),
                      (oracle.digest_f32, v[lo:hi], lo), (oracle.digest_u16, wb[lo:hi], lo)]
        dv = [0, 0, 0, 0]
        for k, r in enumerate(pool.map(lambda a: a[0](a[1], g0 + a[2]), parts)):
            dv[k % 4] = (dv[k % 4] + r) & M64
    t2 = time.perf_counter()
    return t1 - t0, t2 - t1, d, d == dv


def _flat_range(w):
    """The workload's global index range; every workload's pieces cover one
    contiguous range, so the oracle can run it as one flat shard (the digest
    of a concatenation is the sum of the digests, so the table's split does
    not change any result)."""
    lo = min(pc.goff for pc in w.pieces)
    hi = max(pc.goff + pc.n for pc in w.pieces)
    assert hi - lo == w.n
    return lo, hi


def cpu_baseline(cores: int, plan_c5: bool = True, chunk: int = 1 << 22):
    """The oracle (as it stands) on the host cores, per the measurement plan:
    c2, c3 and c4 each timed single-threaded and on all cores over the whole
    workload, and c5 streamed over all of its elements in chunks on all
    cores, with each chunk's oracle compute timed on its own thread (input
    generation is not timed).  One step = the committed step plus the
    verification digests of the written buffers.  Returns the record and the
    oracle's c5 digests of one step from the generated state."""
    from concurrent.futures import ThreadPoolExecutor
    import oracle
    import synth
    from synth import workloads as W
    configs = {}
    with ThreadPoolExecutor(cores) as pool:
        for name in ("c2", "c3", "c4"):
            w = W.ALL[name]()
            lo, hi = _flat_range(w)
            step = w.steps[-1]
            h8 = oracle.resolve_hparams(HP, step)
            p, m, v = synth.state(hi - lo, lo, nthreads=cores)
            g = synth.grad(hi - lo, lo, step, nthreads=cores)
            rec = {"elements": w.n, "step": step}
            for label, th in (("single_thread", 1), ("all_cores", cores)):
                cs, vs, _, ok = _oracle_step(p, m, v, g, lo, h8, th, pool)
                rec[label] = {"threads": th, "commit_s": cs, "verify_s": vs,
                              "elements_per_s": w.n / (cs + vs), "verify_matches_commit": ok}
            configs[name] = rec
            del p, m, v, g
    c5_digests = None
    if plan_c5:
        w = W.c5()
        step = w.steps[-1]
        h8 = oracle.resolve_hparams(HP, step)
        lo, hi = _flat_range(w)

        def one(start):
            n = min(chunk, hi - start)
            p, m, v = synth.state(n, start, nthreads=1)
            g = synth.grad(n, start, step, nthreads=1)
            cs, vs, d, ok = _oracle_step(p, m, v, g, start, h8, 1)
            return cs, vs, d, ok

        t0 = time.perf_counter()
        cs_sum = vs_sum = 0.0
        tot, ok_all, nchunks = [0, 0, 0, 0], True, 0
        with ThreadPoolExecutor(cores) as pool:
            for cs, vs, d, ok in pool.map(one, range(lo, hi, chunk)):
                cs_sum += cs
                vs_sum += vs
                tot = [(a + b) & M64 for a, b in zip(tot, d)]
                ok_all = ok_all and ok
                nchunks += 1
        wall = time.perf_counter() - t0
        c5_digests = tot
        configs["c5"] = {"elements": w.n, "step": step, "chunks": nchunks, "chunk_elements": chunk,
                         "threads": cores, "commit_cpu_s": cs_sum, "verify_cpu_s": vs_sum,
                         "elements_per_s_per_core": w.n / (cs_sum + vs_sum),
                         "elements_per_s_all_cores": w.n * cores / (cs_sum + vs_sum),
                         "wall_s_with_generation": wall, "verify_matches_commit": ok_all,
                         "digests": ["%016x" % x for x in tot],
                         "note": "sum over chunks of each chunk's oracle compute on its own thread; all cores "
                                 "= elements x threads / summed compute seconds"}
    if "c5" in configs:
        value, sample = configs["c5"]["elements_per_s_all_cores"], (
            "all %d elements of c5 (step 18) in %d chunks of %d on %d threads; commit + verification digests; "
            "value = elements x threads / summed per-chunk compute seconds; input generation not timed"
            % (configs["c5"]["elements"], configs["c5"]["chunks"], chunk, cores))
    else:
        value, sample = configs["c4"]["all_cores"]["elements_per_s"], (
            "all %d elements of c4 (step 5) on %d threads, commit + verification digests" % (W.c4().n, cores))
    rec = {"value": value, "unit": "elements/s", "cores": cores, "cpu_model": cpu_model(), "kind": "oracle",
           "sample": sample, "configs": configs}
    return rec, c5_digests


def run_reference(args):
    """The reference arm: the CPU oracle as it stands, on the host cores.
    Each step is one oracle step (commit + verification digests, on all
    cores) over a bounded sample of the workload: its first
    --ref-elements elements; ms_per_step and value are measured on exactly
    those elements."""
    world, rank, _ = dist_env()
    if rank != 0:
        return
    from concurrent.futures import ThreadPoolExecutor
    import oracle
    import synth
    from synth import workloads as W
    w = W.ALL[args.workload]()
    step_t = w.steps[-1]
    lo, hi = _flat_range(w)
    n = min(args.ref_elements, hi - lo)
    cores = os.cpu_count() or 1
    h8 = oracle.resolve_hparams(HP, step_t)
    p, m, v = synth.state(n, lo, nthreads=cores)
    g = synth.grad(n, lo, step_t, nthreads=cores)
    times, ok = [], True
    with ThreadPoolExecutor(cores) as pool:
        for k in range(args.warmup + args.steps):
            cs, vs, _, good = _oracle_step(p, m, v, g, lo, h8, cores, pool)
            ok = ok and good
            if k >= args.warmup:
                times.append(cs + vs)
    t = sum(times) / len(times)
    v_ = n / t
    first = w.pieces[0].name
    sample = ("first %d of the %d elements of %s (from %s on), step %d, committed step + verification digests "
              "on %d threads, %d timed steps" % (n, w.n, w.name, first, step_t, cores, len(times)))
    line = {"impl": "reference", "metric": METRIC, "value": v_, "unit": "elements/s", "n_gpus": world,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1e3 * t, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f32+u64", "data": "synthetic",
            "config": {"workload": "%s: CPU oracle over a bounded sample (%s)" % (w.name, sample), "elements": n,
                       "workload_elements": w.n, "step": step_t},
            "verify_matches_commit": ok,
            "cpu_baseline": {"value": v_, "unit": "elements/s", "cores": cores, "cpu_model": cpu_model(),
                             "kind": "oracle", "sample": sample},
            "e2e": {"value": v_, "unit": "elements/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


def main(argv=None):
    ap = argparse.ArgumentParser(description=__doc__.splitlines()[0])
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=10)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--workload", choices=["c1", "c2", "c3", "c4", "c5"], default="c5")
    ap.add_argument("--schedule", choices=["sequential", "pipelined"], default="sequential",
                    help="sequential: commit, then verify, on one stream; pipelined: the table in --groups groups, "
                         "each group's verification on a second stream beside the next groups' commits")
    ap.add_argument("--groups", type=int, default=12, help="groups of the pipelined schedule")
    ap.add_argument("--commit-grid", type=int, default=0,
                    help="pipelined schedule: CTAs of each commit launch (0: the library's persistent grid)")
    ap.add_argument("--verify-grid", type=int, default=0,
                    help="pipelined schedule: CTAs of each verification launch (0: the library's grid)")
    ap.add_argument("--split", choices=["copy", "model"], default="copy",
                    help="multi-GPU: every rank a full-size copy of the workload (copy, weak scaling) or rank r "
                         "the contiguous range r of the one model's flat parameters (model, strong scaling)")
    ap.add_argument("--e2e-steps", type=int, default=16,
                    help="timed end-to-end steps (each timed region starts with an empty upload pipeline)")
    ap.add_argument("--e2e-groups", type=int, default=12)
    ap.add_argument("--f3-tensors", type=int, default=0,
                    help="next row f3 over the first K tensors of its shard only (0 = all; for profiling)")
    ap.add_argument("--e2e-upload", choices=["sm", "copy"], default="sm",
                    help="end-to-end upload: apc_upload on a few CTAs, or the DMA copy engines")
    ap.add_argument("--e2e-upload-ctas", type=int, default=16)
    ap.add_argument("--e2e-reserved-sms", type=int, default=8)
    ap.add_argument("--ref-elements", type=int, default=1 << 28,
                    help="reference arm: oracle elements per step (a bounded sample of the workload)")
    ap.add_argument("--cpu-plan", choices=["full", "configs"], default="full",
                    help="cpu_baseline: c2-c4 single-thread and all-core, plus c5 streamed over every element "
                         "(full), or c2-c4 only (configs)")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-clocks", action="store_true")
    ap.add_argument("--no-next", action="store_true", help="skip the next-row measurements (f1, f3, f4)")
    ap.add_argument("--replicas", type=int, default=4, help="replica processes of the f4 verification (<= 1: skip)")
    args = ap.parse_args(argv)
    if args.warmup < 3 and args.impl == "ours":
        print("note: at least 3 warm-up steps are required for a valid number", file=sys.stderr)
    if args.impl == "reference":
        run_reference(args)
    else:
        run_gpu(args)


if __name__ == "__main__":
    main()
