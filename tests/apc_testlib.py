"""Shared helpers of the GPU parity tests: device layouts of the workloads,
the streamed CPU oracle over a workload, and sampled comparisons.

Inputs come only from the seeded generator (host or device fill, which are
bit-identical) and expected values only from ``oracle``.
"""
from __future__ import annotations

import os

import numpy as np

import oracle
import synth
from synth import workloads as W

M64 = (1 << 64) - 1
NTHREADS = os.cpu_count() or 1


def gf32(g16: np.ndarray) -> np.ndarray:
    return (g16.astype(np.uint32) << 16).view(np.float32)


class DeviceWorkload:
    """p, m, v (fp32), g, w (bf16 bits) per allocation of a workload, on the
    current CUDA device, filled from the generator by the device fill."""

    def __init__(self, w: W.Workload, grad_step: int, device="cuda"):
        import torch
        self.w = w
        self.alloc_goff = [None] * len(w.allocs)
        for p in w.pieces:
            g0 = p.goff - p.at
            assert self.alloc_goff[p.alloc] in (None, g0)
            self.alloc_goff[p.alloc] = g0
        self.bufs = []
        for a, n in enumerate(w.allocs):
            b = dict(p=torch.empty(n, dtype=torch.float32, device=device),
                     m=torch.empty(n, dtype=torch.float32, device=device),
                     v=torch.empty(n, dtype=torch.float32, device=device),
                     g=torch.empty(n, dtype=torch.int16, device=device),
                     w=torch.empty(n, dtype=torch.int16, device=device))
            self.bufs.append(b)
        self.fill_state()
        self.fill_grad(grad_step)

    def fill_state(self):
        import torch
        s = torch.cuda.current_stream().cuda_stream
        for a, b in enumerate(self.bufs):
            g0, n = self.alloc_goff[a], b["p"].numel()
            synth.fill_dev(synth.P, b["p"].data_ptr(), n, g0, stream=s)
            synth.fill_dev(synth.M, b["m"].data_ptr(), n, g0, stream=s)
            synth.fill_dev(synth.V, b["v"].data_ptr(), n, g0, stream=s)
            b["w"].fill_(0)

    def fill_grad(self, step: int):
        import torch
        s = torch.cuda.current_stream().cuda_stream
        for a, b in enumerate(self.bufs):
            synth.fill_dev(synth.G, b["g"].data_ptr(), b["g"].numel(), self.alloc_goff[a], step=step, stream=s)

    def entries(self):
        import paper_2609_18178_gb300 as apc
        out = []
        for p in self.w.pieces:
            b = self.bufs[p.alloc]
            sl = slice(p.at, p.at + p.n)
            out.append(apc.TensorEntry(b["p"][sl], b["m"][sl], b["v"][sl], b["g"][sl], b["w"][sl], p.goff))
        return out

    def digest_buffers(self):
        import paper_2609_18178_gb300 as apc
        out = []
        for p in self.w.pieces:
            b = self.bufs[p.alloc]
            sl = slice(p.at, p.at + p.n)
            out += apc.state_buffers(b["p"][sl], b["m"][sl], b["v"][sl], b["w"][sl], p.goff)
        return out

    def locate(self, gidx: np.ndarray):
        """(alloc, offset) of global indices."""
        starts = np.array([p.goff for p in self.w.pieces], dtype=np.int64)
        order = np.argsort(starts)
        k = order[np.searchsorted(starts[order], gidx.astype(np.int64), side="right") - 1]
        alloc = np.array([self.w.pieces[i].alloc for i in k])
        off = gidx.astype(np.int64) - starts[k] + np.array([self.w.pieces[i].at for i in k])
        return alloc, off

    def gather(self, gidx: np.ndarray):
        """Device values (p, m, v as uint32 bits, w as uint16) at global indices."""
        import torch
        alloc, off = self.locate(gidx)
        res = {k: np.empty(len(gidx), dtype=np.uint32 if k != "w" else np.uint16) for k in "pmvw"}
        for a in np.unique(alloc):
            sel = np.nonzero(alloc == a)[0]
            idx = torch.from_numpy(off[sel]).to(self.bufs[a]["p"].device)
            for k in "pmv":
                res[k][sel] = self.bufs[a][k].index_select(0, idx).cpu().numpy().view(np.uint32)
            res["w"][sel] = self.bufs[a]["w"].index_select(0, idx).cpu().numpy().view(np.uint16)
        return res


def oracle_at(gidx: np.ndarray, step: int, hp=None):
    """Oracle outputs of one step from the generated state at global indices."""
    hp = hp or oracle.DEFAULT_HP
    p = synth.fill_at(synth.P, gidx)
    m = synth.fill_at(synth.M, gidx)
    v = synth.fill_at(synth.V, gidx)
    g = synth.fill_at(synth.G, gidx, step=step)
    w = oracle.adamw(p, m, v, g, oracle.resolve_hparams(hp, step))
    return dict(p=p.view(np.uint32), m=m.view(np.uint32), v=v.view(np.uint32), w=w)


def oracle_workload_digest(w: W.Workload, step: int, hp=None, chunk: int = 1 << 22, workers: int | None = None,
                           inspect=None):
    """The four digests of one step over a workload from the generated state,
    streamed through the oracle chunk by chunk (host memory stays bounded).

    Chunks run concurrently on ``workers`` threads (default: every host
    core), each generating its inputs and running the oracle single-threaded;
    the oracle and the generator are C calls that release the GIL.  The
    digests of the chunks are added mod 2^64, which is the digest of their
    concatenation.  ``inspect(piece, start, outputs)``, if given, is called
    (on a worker thread) for every chunk of every piece with
    ``outputs = dict(p, m, v, w)`` holding the oracle's written bits of
    elements [start, start + n) of that piece, so that a test can compare
    whole tensors element by element on the way."""
    from concurrent.futures import ThreadPoolExecutor
    hp = hp or oracle.DEFAULT_HP
    h8 = oracle.resolve_hparams(hp, step)
    jobs = [(pc, s) for pc in w.pieces for s in range(0, pc.n, chunk)]

    def run(job):
        pc, s = job
        n = min(chunk, pc.n - s)
        g0 = pc.goff + s
        p, m, v = synth.state(n, g0, nthreads=1)
        g = synth.grad(n, g0, step, nthreads=1)
        wb, d = oracle.commit(p, m, v, g, g0, h8, nthreads=1)
        if inspect is not None:
            inspect(pc, s, dict(p=p.view(np.uint32), m=m.view(np.uint32), v=v.view(np.uint32), w=wb))
        return d

    tot = [0, 0, 0, 0]
    with ThreadPoolExecutor(workers or NTHREADS) as ex:
        for d in ex.map(run, jobs):
            tot = [(a + b) & M64 for a, b in zip(tot, d)]
    return tot


def sample_indices(w: W.Workload, k: int, seed: int) -> np.ndarray:
    """Random global indices plus the first/last elements of every piece and
    the elements around 2^32."""
    rng = np.random.default_rng(seed)
    idx = []
    for pc in w.pieces:
        idx += [pc.goff, pc.goff + pc.n - 1, pc.goff + min(7, pc.n - 1), pc.goff + max(0, pc.n - 8)]
    lo, hi = min(p.goff for p in w.pieces), max(p.goff + p.n for p in w.pieces)
    for x in ((1 << 32) - 2, (1 << 32) - 1, 1 << 32, (1 << 32) + 1):
        if lo <= x < hi:
            idx.append(x)
    total = w.n
    starts = np.cumsum([0] + [p.n for p in w.pieces])
    r = rng.integers(0, total, size=k)
    j = np.searchsorted(starts, r, side="right") - 1
    idx += [w.pieces[a].goff + int(r[i] - starts[a]) for i, a in enumerate(j)]
    return np.unique(np.array(idx, dtype=np.uint64))


class DeviceWorkloadBF16:
    """bf16 p, m, v and g per allocation of a workload on the current CUDA
    device, filled from the generator by the device fill."""

    def __init__(self, w: W.Workload, grad_step: int, device="cuda"):
        import torch
        self.w = w
        self.alloc_goff = [None] * len(w.allocs)
        for p in w.pieces:
            self.alloc_goff[p.alloc] = p.goff - p.at
        s = torch.cuda.current_stream().cuda_stream
        self.bufs = []
        for a, n in enumerate(w.allocs):
            b = {k: torch.empty(n, dtype=torch.int16, device=device) for k in "pmvg"}
            g0 = self.alloc_goff[a]
            synth.fill_dev(synth.P16, b["p"].data_ptr(), n, g0, stream=s)
            synth.fill_dev(synth.M16, b["m"].data_ptr(), n, g0, stream=s)
            synth.fill_dev(synth.V16, b["v"].data_ptr(), n, g0, stream=s)
            synth.fill_dev(synth.G, b["g"].data_ptr(), n, g0, step=grad_step, stream=s)
            self.bufs.append(b)

    def entries(self):
        import paper_2609_18178_gb300 as apc
        out = []
        for p in self.w.pieces:
            b = self.bufs[p.alloc]
            sl = slice(p.at, p.at + p.n)
            out.append(apc.TensorEntryBF16(b["p"][sl], b["m"][sl], b["v"][sl], b["g"][sl], p.goff))
        return out

    def digest_buffers(self):
        import paper_2609_18178_gb300 as apc
        out = []
        for p in self.w.pieces:
            b = self.bufs[p.alloc]
            sl = slice(p.at, p.at + p.n)
            out += apc.state_buffers_bf16(b["p"][sl], b["m"][sl], b["v"][sl], p.goff)
        return out

    def gather(self, gidx: np.ndarray):
        import torch
        starts = np.array([p.goff for p in self.w.pieces], dtype=np.int64)
        k = np.searchsorted(starts, gidx.astype(np.int64), side="right") - 1
        alloc = np.array([self.w.pieces[i].alloc for i in k])
        off = gidx.astype(np.int64) - starts[k] + np.array([self.w.pieces[i].at for i in k])
        res = {key: np.empty(len(gidx), dtype=np.uint16) for key in "pmv"}
        for a in np.unique(alloc):
            sel = np.nonzero(alloc == a)[0]
            idx = torch.from_numpy(off[sel]).to(self.bufs[a]["p"].device)
            for key in "pmv":
                res[key][sel] = self.bufs[a][key].index_select(0, idx).cpu().numpy().view(np.uint16)
        return res


def oracle_at_bf16(gidx: np.ndarray, step: int, hp=None):
    """Oracle outputs of one bf16-state step from the generated state at global indices."""
    hp = hp or oracle.DEFAULT_HP
    p = synth.fill_at(synth.P16, gidx)
    m = synth.fill_at(synth.M16, gidx)
    v = synth.fill_at(synth.V16, gidx)
    g = synth.fill_at(synth.G, gidx, step=step)
    oracle.adamw_bf16(p, m, v, g, oracle.resolve_hparams(hp, step))
    return dict(p=p, m=m, v=v)


def oracle_workload_digest_bf16(w: W.Workload, step: int, lo: int, hi: int, hp=None, chunk: int = 1 << 24):
    """The three bf16-state digests of one step over the part [lo, hi) of a
    workload's global range, streamed through the oracle."""
    hp = hp or oracle.DEFAULT_HP
    h8 = oracle.resolve_hparams(hp, step)
    tot = [0, 0, 0]
    for s in range(lo, hi, chunk):
        n = min(chunk, hi - s)
        p, m, v = synth.state_bf16(n, s, nthreads=NTHREADS)
        g = synth.grad(n, s, step, nthreads=NTHREADS)
        d = oracle.commit_bf16(p, m, v, g, s, h8)
        tot = [(a + b) & M64 for a, b in zip(tot, d)]
    return tot
