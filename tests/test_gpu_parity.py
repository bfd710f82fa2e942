"""GPU parity of the CUDA path (through the C ABI) against the CPU oracle.

Bar: every written float and bf16 word bit-identical (0 ulp) and every digest
equal.  Small cases compare every element; the paper-sized workloads compare
full digests against the streamed oracle where the host can regenerate them
in seconds, and sampled elements plus digest properties at the largest size,
in the same launch configuration the benchmark times.
"""
import numpy as np
import pytest

import oracle
import synth
from synth import workloads as W

from apc_testlib import (M64, DeviceWorkload, gf32, oracle_at, oracle_workload_digest, sample_indices)

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

if not torch.cuda.is_available():  # the CUDA path has no fallback: without a GPU these tests cannot run
    pytest.skip("no CUDA device", allow_module_level=True)

import paper_2609_18178_gb300 as apc  # noqa: E402

HP = oracle.DEFAULT_HP


def dev(a):
    t = torch.from_numpy(np.ascontiguousarray(a))
    if t.dtype == torch.uint16:
        t = t.view(torch.int16)
    return t.cuda()


def host(t, dt):
    return t.cpu().numpy().view(dt)


def run_small(tensors, step, hp=HP):
    """tensors: list of dict(p, m, v, g numpy, goff).  Runs the CUDA path and
    the oracle on copies; returns (device results, oracle results)."""
    entries, devs = [], []
    for t in tensors:
        d = dict(p=dev(t["p"]), m=dev(t["m"]), v=dev(t["v"]), g=dev(t["g"]),
                 w=torch.zeros(t["p"].size, dtype=torch.int16, device="cuda"))
        devs.append(d)
        entries.append(apc.TensorEntry(d["p"], d["m"], d["v"], d["g"], d["w"], t["goff"]))
    out = apc.commit_step(entries, step, hp)
    torch.cuda.synchronize()
    h8 = oracle.resolve_hparams(hp, step)
    ref = [dict(p=t["p"].copy(), m=t["m"].copy(), v=t["v"].copy(), g=t["g"], goff=t["goff"]) for t in tensors]
    ws, dref = oracle.commit_table(ref, h8)
    for r, wv in zip(ref, ws):
        r["w"] = wv
    return devs, apc.digests_to_host(out), ref, dref


def assert_same(devs, dgot, ref, dref):
    for d, r in zip(devs, ref):
        for k in "pmv":
            a, b = host(d[k], np.uint32), r[k].view(np.uint32)
            bad = np.nonzero(a != b)[0]
            assert bad.size == 0, "%s differs at %s: %s vs %s" % (k, bad[:5], a[bad[:5]], b[bad[:5]])
        a, b = host(d["w"], np.uint16), r["w"]
        assert np.array_equal(a, b), "w differs"
    assert dgot == dref, "digests differ"


def gen(n, goff, step, seed_shift=0):
    p, m, v = synth.state(n, goff)
    return dict(p=p, m=m, v=v, g=synth.grad(n, goff, step), goff=goff)


def test_c1_chained_three_steps():
    w = W.c1()
    n = w.n
    t = gen(n, 0, 1)
    state = dict(p=t["p"], m=t["m"], v=t["v"])
    d = dict(p=dev(state["p"]), m=dev(state["m"]), v=dev(state["v"]),
             w=torch.zeros(n, dtype=torch.int16, device="cuda"))
    for step in (1, 2, 3):
        g = synth.grad(n, 0, step)
        d["g"] = dev(g)
        out = apc.commit_step([apc.TensorEntry(d["p"], d["m"], d["v"], d["g"], d["w"], 0)], step, HP)
        torch.cuda.synchronize()
        wv, dref = oracle.commit(state["p"], state["m"], state["v"], g, 0, oracle.resolve_hparams(HP, step))
        for k in "pmv":
            assert np.array_equal(host(d[k], np.uint32), state[k].view(np.uint32)), (step, k)
        assert np.array_equal(host(d["w"], np.uint16), wv)
        assert apc.digests_to_host(out) == dref
        ver = apc.digest(apc.state_buffers(d["p"], d["m"], d["v"], d["w"], 0), 4)
        assert apc.digests_to_host(ver) == dref


# Elements per tile of the commit kernel (19 consumer warps x 32 threads x 2 groups of 4).
COMMIT_TILE = 4864


@pytest.mark.parametrize("n", list(range(1, 65)) + [127, 129, 4095, 4096, 4097, 8191, 8199, 100003] +
                         [k * COMMIT_TILE + d for k in (1, 2) for d in (-8, -1, 0, 1, 8)])
def test_small_sizes(n):
    goff = (1 << 32) - n // 2 - 3
    assert_same(*run_small([gen(n, goff, 2)], 2))


@pytest.mark.parametrize("goff", [0, 5, (1 << 32) - 1, (1 << 32) + 77, M64 - 70000, (1 << 40) + 3])
def test_global_offsets(goff):
    n = 60000 if goff < M64 - 70000 else 70000
    t = gen(n, 0, 3)
    t["goff"] = goff
    assert_same(*run_small([t], 3))


@pytest.mark.parametrize("shift", range(1, 8))
def test_uniform_misalignment_uses_head(shift):
    """All five buffers start `shift` elements past a 16-byte boundary."""
    n = 20000 + shift
    t = gen(n + shift, 100, 4)
    base = dict(p=dev(t["p"]), m=dev(t["m"]), v=dev(t["v"]), g=dev(t["g"]),
                w=torch.zeros(n + shift, dtype=torch.int16, device="cuda"))
    sl = slice(shift, shift + n)
    out = apc.commit_step([apc.TensorEntry(base["p"][sl], base["m"][sl], base["v"][sl], base["g"][sl],
                                           base["w"][sl], 100 + shift)], 4, HP)
    torch.cuda.synchronize()
    ref = dict(p=t["p"][sl].copy(), m=t["m"][sl].copy(), v=t["v"][sl].copy())
    wv, dref = oracle.commit(ref["p"], ref["m"], ref["v"], np.ascontiguousarray(t["g"][sl]), 100 + shift,
                             oracle.resolve_hparams(HP, 4))
    for k in "pmv":
        got = host(base[k], np.uint32)
        assert np.array_equal(got[sl], ref[k].view(np.uint32))
        assert np.array_equal(got[:shift], t[k][:shift].view(np.uint32))  # untouched before the slice
    gw = host(base["w"], np.uint16)
    assert np.array_equal(gw[sl], wv) and not gw[:shift].any()
    assert apc.digests_to_host(out) == dref


@pytest.mark.parametrize("pshift,gshift", [(1, 0), (0, 3), (2, 1), (3, 5)])
def test_mutual_misalignment_runs_scalar(pshift, gshift):
    n = 9000
    t = gen(n + 8, 0, 5)
    P, Mm, V = dev(t["p"]), dev(t["m"]), dev(t["v"])
    G = dev(t["g"])
    Wt = torch.zeros(n + 8, dtype=torch.int16, device="cuda")
    ps, gs = slice(pshift, pshift + n), slice(gshift, gshift + n)
    out = apc.commit_step([apc.TensorEntry(P[ps], Mm[ps], V[ps], G[gs], Wt[gs], 7)], 5, HP)
    torch.cuda.synchronize()
    ref = dict(p=t["p"][ps].copy(), m=t["m"][ps].copy(), v=t["v"][ps].copy())
    wv, dref = oracle.commit(ref["p"], ref["m"], ref["v"], np.ascontiguousarray(t["g"][gs]), 7,
                             oracle.resolve_hparams(HP, 5))
    assert np.array_equal(host(P, np.uint32)[ps], ref["p"].view(np.uint32))
    assert np.array_equal(host(Mm, np.uint32)[ps], ref["m"].view(np.uint32))
    assert np.array_equal(host(V, np.uint32)[ps], ref["v"].view(np.uint32))
    assert np.array_equal(host(Wt, np.uint16)[gs], wv)
    assert apc.digests_to_host(out) == dref


def test_many_tensors_several_launches():
    """1200 ragged tensors (more than one launch's table capacity), as views
    with gaps into shared allocations."""
    rng = np.random.default_rng(11)
    sizes = rng.integers(1, 3000, size=1200)
    tensors, off = [], (1 << 32) - 1_000_000
    for n in sizes:
        tensors.append(gen(int(n), off, 6))
        off += int(n)
    assert_same(*run_small(tensors, 6))


def test_empty_table_and_zero_length_entries():
    out = torch.full((4,), 123, dtype=torch.int64, device="cuda")
    apc.commit_step([], 1, HP, out=out)
    torch.cuda.synchronize()
    assert apc.digests_to_host(out) == [0, 0, 0, 0]
    t = gen(1000, 50, 1)
    devs, dgot, ref, dref = run_small([t], 1)
    d = devs[0]
    entries = [apc.TensorEntry(0, 0, 0, 0, 0, 0, n=0),
               apc.TensorEntry(d["p"], d["m"], d["v"], d["g"], d["w"], 50, n=0)]
    apc.commit_step(entries, 1, HP, out=out)
    torch.cuda.synchronize()
    assert apc.digests_to_host(out) == [0, 0, 0, 0]
    # the data were not touched by the zero-length call
    assert np.array_equal(host(d["p"], np.uint32), ref[0]["p"].view(np.uint32))


def test_prepared_tables_match_the_oracle_over_chained_steps():
    """A table marshalled once (prepare_table / prepare_buffers) and reused
    for chained steps gives the oracle's state and digests at every step."""
    tensors = [gen(n, off, 1) for n, off in ((4999, 0), (8, 4999), (20011, 5007))]
    entries, devs = [], []
    for t in tensors:
        d = dict(p=dev(t["p"]), m=dev(t["m"]), v=dev(t["v"]), g=dev(t["g"]),
                 w=torch.zeros(t["p"].size, dtype=torch.int16, device="cuda"))
        devs.append(d)
        entries.append(apc.TensorEntry(d["p"], d["m"], d["v"], d["g"], d["w"], t["goff"]))
    tab = apc.prepare_table(entries)
    vtab = apc.prepare_buffers([b for e in entries for b in apc.state_buffers(e.p, e.m, e.v, e.w, e.global_offset)])
    ref = [dict(p=t["p"].copy(), m=t["m"].copy(), v=t["v"].copy(), g=t["g"], goff=t["goff"]) for t in tensors]
    for step in (1, 2, 3):
        got = apc.digests_to_host(apc.commit_step(tab, step, HP))
        ver = apc.digests_to_host(apc.digest(vtab, 4))
        ws, dref = oracle.commit_table(ref, oracle.resolve_hparams(HP, step))
        for r, wv in zip(ref, ws):
            r["w"] = wv
        assert got == dref and ver == dref
        assert_same(devs, got, ref, dref)


def test_guard_bands_untouched():
    """Canary words around every buffer stay intact (bounds of the vector
    head, body and tail paths)."""
    pad = 1024
    for n, shift in ((37, 3), (4096 + 5, 1), (12345, 0)):
        t = gen(n, 1000, 2)
        bufs = {}
        for k, dt in (("p", np.float32), ("m", np.float32), ("v", np.float32), ("g", np.uint16), ("w", np.uint16)):
            a = np.full(n + 2 * pad, 0x5A5A if dt == np.uint16 else np.float32(7.25), dtype=dt)
            if k != "w":
                a[pad:pad + n] = t[k]
            bufs[k] = dev(a)
        sl = slice(pad, pad + n)
        apc.commit_step([apc.TensorEntry(bufs["p"][sl], bufs["m"][sl], bufs["v"][sl], bufs["g"][sl],
                                         bufs["w"][sl], 1000)], 2, HP)
        torch.cuda.synchronize()
        for k in "pmv":
            a = host(bufs[k], np.float32)
            assert np.all(a[:pad] == np.float32(7.25)) and np.all(a[pad + n:] == np.float32(7.25))
        for k in "gw":
            a = host(bufs[k], np.uint16)
            assert np.all(a[:pad] == 0x5A5A) and np.all(a[pad + n:] == 0x5A5A)


def test_digest_of_arbitrary_buffers():
    rng = np.random.default_rng(12)
    bufs, want, keep = [], [0] * 8, []
    for i in range(1100):                       # more than one launch's capacity
        n = int(rng.integers(0, 700))
        goff = int(rng.integers(0, 1 << 34))
        slot = int(rng.integers(0, 8))
        f32 = bool(rng.integers(0, 2))
        shift = int(rng.integers(0, 8))
        if f32:
            a = rng.integers(0, 2**32, size=n + shift, dtype=np.uint64).astype(np.uint32)
            t = torch.from_numpy(a.view(np.int32)).cuda()
            want[slot] = (want[slot] + oracle.digest_f32(a[shift:], goff)) & M64
        else:
            a = rng.integers(0, 2**16, size=n + shift, dtype=np.uint64).astype(np.uint16)
            t = torch.from_numpy(a.view(np.int16)).cuda()
            want[slot] = (want[slot] + oracle.digest_u16(a[shift:], goff)) & M64
        keep.append(t)
        bufs.append(apc.BufferEntry(t[shift:], slot, goff, apc.F32 if f32 else apc.BF16))
    out = apc.digest(bufs, 8)
    assert apc.digests_to_host(out) == want


# Elements per tile of the verification kernel (1024 threads x 2 vectors of 8)
# and of the guard kernel (1024 x 4): every tile of a buffer but its last runs
# without bounds checks.
DIGEST_TILE = 16384
COUNT_TILE = 32768


@pytest.mark.parametrize("limit", [None, 1, 5])
def test_digest_buffers_at_tile_boundaries(monkeypatch, limit):
    """Buffers whose vector bodies end exactly on, just before and just after
    a tile boundary, with and without a scalar head, on the default grid and
    on grids of 1 and 5 CTAs (whose contiguous tile runs then start and end
    inside buffers): every slot's digest equals the oracle's."""
    if limit is None:
        monkeypatch.delenv("APC_GRID_LIMIT", raising=False)
    else:
        monkeypatch.setenv("APC_GRID_LIMIT", str(limit))
    rng = np.random.default_rng(33)
    bufs, each, keep = [], [], []
    sizes = [k * DIGEST_TILE + d for k in (1, 2, 3) for d in (-8, -1, 0, 1, 7, 8, 9)] + [5 * DIGEST_TILE + 8 * 1024]
    for i, n in enumerate(sizes):
        for f32 in (True, False):
            shift = int(rng.integers(1, 8)) if i % 2 else 0   # a nonzero shift gives a scalar head
            goff = int(rng.integers(0, 1 << 33))
            slot = (2 * i + f32) % 4
            if f32:
                a = rng.integers(0, 2**32, size=n + shift, dtype=np.uint64).astype(np.uint32)
                t = torch.from_numpy(a.view(np.int32)).cuda()
                each.append((slot, oracle.digest_f32(a[shift:], goff)))
            else:
                a = rng.integers(0, 2**16, size=n + shift, dtype=np.uint64).astype(np.uint16)
                t = torch.from_numpy(a.view(np.int16)).cuda()
                each.append((slot, oracle.digest_u16(a[shift:], goff)))
            keep.append(t)
            bufs.append(apc.BufferEntry(t[shift:], slot, goff, apc.F32 if f32 else apc.BF16))
    want = [0] * 4
    for slot, d in each:
        want[slot] = (want[slot] + d) & M64
    assert apc.digests_to_host(apc.digest(bufs, 4)) == want
    # each buffer alone, so that no wrong term hides behind another buffer's in the same slot
    for b, (slot, d) in zip(bufs, each):
        alone = apc.BufferEntry(b.data, 0, b.global_offset, b.dtype)
        assert apc.digests_to_host(apc.digest([alone], 1))[0] == d, (b.data.numel(), b.dtype)


def test_invalid_arguments_are_rejected():
    t = gen(64, 0, 1)
    d = dict(p=dev(t["p"]), m=dev(t["m"]), v=dev(t["v"]), g=dev(t["g"]),
             w=torch.zeros(64, dtype=torch.int16, device="cuda"))
    e = apc.TensorEntry(d["p"], d["m"], d["v"], d["g"], d["w"], 0)
    with pytest.raises(apc.ApcError) as ei:
        apc.commit_step([e], 0, HP)
    assert ei.value.status == 1
    with pytest.raises(apc.ApcError) as ei:
        apc.commit_step([e, e], 1, HP)          # the same outputs twice overlap
    assert ei.value.status == 1
    with pytest.raises(apc.ApcError) as ei:
        apc.commit_step([apc.TensorEntry(d["p"].data_ptr() + 2, d["m"], d["v"], d["g"], d["w"], 0, n=8)], 1, HP)
    assert ei.value.status == 2
    with pytest.raises(apc.ApcError) as ei:
        apc.commit_step([apc.TensorEntry(d["p"], d["m"], d["v"], d["g"], d["w"], M64 - 10)], 1, HP)
    assert ei.value.status == 3
    # nothing ran: the state is the generated one
    assert np.array_equal(host(d["p"], np.uint32), t["p"].view(np.uint32))


def check_sampled(dw: DeviceWorkload, step: int, k: int, seed: int):
    idx = sample_indices(dw.w, k, seed)
    got = dw.gather(idx)
    ref = oracle_at(idx, step)
    for key in "pmvw":
        bad = np.nonzero(got[key] != ref[key])[0]
        assert bad.size == 0, "%s differs at global %s" % (key, idx[bad[:5]])


@pytest.mark.parametrize("step", [1, 1000])
def test_c2_full_size(step):
    """Mistral-7B MLP unit, 176,160,768 elements, steps 1 and 1000 from the
    generated state: full digests against the streamed oracle and sampled
    elements bit for bit."""
    w = W.c2()
    dw = DeviceWorkload(w, step)
    out = apc.commit_step(dw.entries(), step, HP)
    got = apc.digests_to_host(out)
    check_sampled(dw, step, 100000, step)
    assert got == oracle_workload_digest(w, step)
    assert apc.digests_to_host(apc.digest(dw.digest_buffers(), 4)) == got
    del dw
    torch.cuda.empty_cache()


def test_c3_full_size():
    w = W.c3()
    dw = DeviceWorkload(w, 10)
    got = apc.digests_to_host(apc.commit_step(dw.entries(), 10, HP))
    check_sampled(dw, 10, 100000, 3)
    assert got == oracle_workload_digest(w, 10)
    del dw
    torch.cuda.empty_cache()


def test_c4_rank_shard_pieces_equal_one_entry():
    """Rank 9 of 16 (crosses 2^32): the 21-piece table and the single entry
    give identical bits and digests, equal to the streamed oracle; the verify
    pass reproduces the fused digests."""
    wp, w1 = W.c4(), W.c4(one_entry=True)
    a = DeviceWorkload(wp, 5)
    da = apc.digests_to_host(apc.commit_step(a.entries(), 5, HP))
    check_sampled(a, 5, 100000, 4)
    pa = a.bufs[0]["p"].clone()
    del a
    b = DeviceWorkload(w1, 5)
    db = apc.digests_to_host(apc.commit_step(b.entries(), 5, HP))
    assert torch.equal(pa.view(torch.int32), b.bufs[0]["p"].view(torch.int32))
    assert da == db
    assert apc.digests_to_host(apc.digest(b.digest_buffers(), 4)) == db
    del pa, b
    torch.cuda.empty_cache()
    assert da == oracle_workload_digest(wp, 5)


# Whole tensors of every shape class of Mistral-7B, compared element by
# element on the way through the streamed oracle of the full model.
C5_WHOLE_TENSORS = ("embed_tokens", "layers.13.q_proj", "layers.13.k_proj", "layers.20.down_proj",
                    "layers.31.post_attention_layernorm", "norm", "lm_head")


def test_c5_full_model_bench_configuration():
    """The benchmark's workload: all 291 Mistral-7B tensors (7,248,023,552
    elements) in separate allocations, step 18, the same table and launch
    configuration as bench.py.

    The whole state is checked against the oracle: the four digests of
    p', m', v', w equal those of the oracle streamed over every element of
    the model (the bitwise rank-state check of Sections IV-F/IV-G over the
    W, M, V of Section III-A, Eq. 2), and whole tensors of each shape class
    (embedding, q, k, down projections, both RMSNorm kinds, lm_head) equal it
    bit for bit.  The verify pass equals the fused digests, and the 16 rank
    shards' digests sum to the whole (concatenation)."""
    import threading
    import time
    w = W.c5()
    free, total = torch.cuda.mem_get_info()
    if free < 130 * (1 << 30):
        pytest.skip("needs ~120 GB of free device memory")
    dw = DeviceWorkload(w, 18)
    got = apc.digests_to_host(apc.commit_step(dw.entries(), 18, HP))
    check_sampled(dw, 18, 200000, 5)
    assert apc.digests_to_host(apc.digest(dw.digest_buffers(), 4)) == got
    total = [0, 0, 0, 0]
    for r in range(16):
        lo, hi = W.rank_range(r, 16)
        bufs = []
        for pc in w.pieces:
            a, b = max(pc.goff, lo), min(pc.goff + pc.n, hi)
            if a < b:
                B = dw.bufs[pc.alloc]
                sl = slice(a - pc.goff, b - pc.goff)
                bufs += apc.state_buffers(B["p"][sl], B["m"][sl], B["v"][sl], B["w"][sl], a)
        d = apc.digests_to_host(apc.digest(bufs, 4))
        total = [(x + y) & M64 for x, y in zip(total, d)]
    assert total == got
    torch.cuda.synchronize()

    names = set(C5_WHOLE_TENSORS)
    assert names <= {pc.name for pc in w.pieces}
    compared, bad, lock = {}, [], threading.Lock()

    def inspect(pc, start, ref):
        if pc.name not in names:
            return
        B = dw.bufs[pc.alloc]
        n = len(ref["w"])
        sl = slice(pc.at + start, pc.at + start + n)
        for k in "pmv":
            dev_bits = B[k][sl].cpu().numpy().view(np.uint32)
            if not np.array_equal(dev_bits, ref[k]):
                with lock:
                    bad.append((pc.name, k, start, int(np.count_nonzero(dev_bits != ref[k]))))
        if not np.array_equal(B["w"][sl].cpu().numpy().view(np.uint16), ref["w"]):
            with lock:
                bad.append((pc.name, "w", start))
        with lock:
            compared[pc.name] = compared.get(pc.name, 0) + n

    t0 = time.perf_counter()
    want = oracle_workload_digest(w, 18, inspect=inspect)
    print("c5 oracle stream: %d elements in %.1f s" % (w.n, time.perf_counter() - t0))
    assert not bad, bad[:5]
    assert compared == {pc.name: pc.n for pc in w.pieces if pc.name in names}
    assert got == want
    del dw
    torch.cuda.empty_cache()


def test_repeat_runs_identical():
    w = W.c3()
    res = []
    for _ in range(3):
        dw = DeviceWorkload(w, 10)
        res.append(apc.digests_to_host(apc.commit_step(dw.entries(), 10, HP)))
        del dw
    assert res[0] == res[1] == res[2]
    torch.cuda.empty_cache()


@pytest.mark.parametrize("limit", [None, 1, 7, 64])
def test_grid_size_does_not_change_results(monkeypatch, limit):
    """The same step on persistent grids of 1, 7, 64 CTAs and the default
    (APC_GRID_LIMIT caps the grid): outputs and digests equal the oracle's,
    and so does the verification digest on the same grid."""
    if limit is None:
        monkeypatch.delenv("APC_GRID_LIMIT", raising=False)
    else:
        monkeypatch.setenv("APC_GRID_LIMIT", str(limit))
    tensors = [gen(n, off, 4) for n, off in ((600_001, (1 << 32) - 300_000), (5, 900_000), (448_570, 1_000_000))]
    devs, dgot, ref, dref = run_small(tensors, 4)
    assert_same(devs, dgot, ref, dref)
    bufs = [b for d, t in zip(devs, tensors) for b in apc.state_buffers(d["p"], d["m"], d["v"], d["w"], t["goff"])]
    assert apc.digests_to_host(apc.digest(bufs, 4)) == dref


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_single_bit_flip_changes_digest_by_its_term(dtype):
    """A bit flipped in device memory (through a host copy) changes the
    digest by exactly splitmix64(new key) - splitmix64(old key) mod 2^64,
    for every bit position of the word."""
    rng = np.random.default_rng(21)
    n, goff = 10_007, (1 << 32) - 5_000
    if dtype == "f32":
        udt, sdt, bits, kind = np.uint32, np.int32, 32, apc.F32
    else:
        udt, sdt, bits, kind = np.uint16, np.int16, 16, apc.BF16
    a = rng.integers(0, 1 << bits, size=n, dtype=np.uint64).astype(udt)
    t = torch.from_numpy(a.view(sdt)).cuda()
    buf = [apc.BufferEntry(t, 0, goff, kind)]
    base = apc.digests_to_host(apc.digest(buf, 1))[0]
    assert base == (oracle.digest_f32(a, goff) if dtype == "f32" else oracle.digest_u16(a, goff))
    for b in range(bits):
        i = int(rng.integers(0, n))
        old = int(a[i])
        new = old ^ (1 << b)
        flipped = a.copy()
        flipped[i] = new
        t.copy_(torch.from_numpy(flipped.view(sdt)))          # the flip reaches HBM through a host copy
        got = apc.digests_to_host(apc.digest(buf, 1))[0]
        key = ((goff + i) & 0xFFFFFFFF) << 32
        delta = (oracle.splitmix64(key | new) - oracle.splitmix64(key | old)) & M64
        assert delta != 0 and got == (base + delta) & M64, (b, i)
    t.copy_(torch.from_numpy(a.view(sdt)))
    assert apc.digests_to_host(apc.digest(buf, 1))[0] == base


def test_bounded_wait_gives_up_and_context_stays_usable():
    """A kernel wait that nothing completes expires (about 50 ms and 2^20
    polls), records APC_ETIMEOUT, and the next committed step still runs
    bit-exact."""
    assert apc.device_status() == 0
    apc.selftest_wait_timeout(50_000_000)
    assert apc.device_status() == 5
    assert apc.device_status() == 0          # reading clears the word
    assert_same(*run_small([gen(5000, 123, 2)], 2))
    assert apc.device_status() == 0


def adversarial(n, seed):
    """Generated state with blocks of edge values: v = 0 with g = 0 (den =
    eps), denormal moments, large and tiny gradients, tiny and signed-zero
    parameters, negative-zero moments."""
    rng = np.random.default_rng(seed)
    t = gen(n, seed * n, seed + 1)
    p, m, v, g = t["p"], t["m"], t["v"], t["g"]
    k = n // 8
    v[:k] = 0.0
    g[:k] = 0
    m[k:2 * k] = (rng.standard_normal(k) * 1e-38).astype(np.float32)
    v[k:2 * k] = np.abs(rng.standard_normal(k) * 1e-41).astype(np.float32)
    g[2 * k:3 * k] = ((rng.standard_normal(k).astype(np.float32) * np.float32(10.0)).view(np.uint32) >> 16)
    g[3 * k:4 * k] = ((rng.standard_normal(k).astype(np.float32) * np.float32(1e-12)).view(np.uint32) >> 16)
    p[4 * k:5 * k] = (rng.standard_normal(k) * 1e-30).astype(np.float32)
    p[5 * k:5 * k + 64] = np.float32(-0.0)
    m[5 * k + 64:5 * k + 128] = np.float32(-0.0)
    g[5 * k + 128:5 * k + 192] = 0x8000          # bf16 -0
    return t


@pytest.mark.parametrize("hp", [HP, dict(HP, lr=0.0), dict(HP, beta1=0.0), dict(HP, weight_decay=0.0),
                                dict(lr=1e-2, beta1=0.5, beta2=0.999, eps=1e-6, weight_decay=0.01)])
@pytest.mark.parametrize("step", [1, 7, 1000])
def test_hyperparameters_and_edge_values(hp, step):
    assert_same(*run_small([adversarial(40000, step), adversarial(333, step + 1)], step, hp))


F32_NAN = np.array([0x7FC00000, 0xFFC00000, 0x7F800001, 0x7FFFFFFF], np.uint32).view(np.float32)
BF16_NAN = np.array([0x7FC0, 0xFFC0, 0x7F81, 0xFFFF], np.uint16)


def nonfinite(n, seed):
    """Generated state with non-finite inputs: blocks of infinite and NaN
    gradients, parameters and moments and of negative second moments (whose
    square root is NaN), then single non-finite values scattered over the
    rest, so that packed pairs and vectors mix NaN and finite lanes."""
    rng = np.random.default_rng(seed)
    t = gen(n, seed * n, seed + 1)
    p, m, v, g = t["p"], t["m"], t["v"], t["g"]
    k = n // 12
    inf = np.array([np.inf, -np.inf], np.float32)
    g[:k] = rng.choice(np.array([0x7F80, 0xFF80], np.uint16), k)
    g[k:2 * k] = rng.choice(BF16_NAN, k)
    p[2 * k:3 * k] = rng.choice(inf, k)
    p[3 * k:4 * k] = rng.choice(F32_NAN, k)
    m[4 * k:5 * k] = rng.choice(inf, k)
    m[5 * k:6 * k] = rng.choice(F32_NAN, k)
    v[6 * k:7 * k] = np.inf
    v[7 * k:8 * k] = rng.choice(F32_NAN, k)
    v[8 * k:9 * k] = -np.abs(v[8 * k:9 * k]) - np.float32(1e-3)
    rest = np.arange(9 * k, n)
    for a, pool in ((p, np.concatenate([inf, F32_NAN])), (m, np.concatenate([inf, F32_NAN])),
                    (v, np.concatenate([inf[:1], F32_NAN])), (g, np.concatenate([np.array([0x7F80, 0xFF80],
                                                                                     np.uint16), BF16_NAN]))):
        at = rest[rng.random(rest.size) < 0.03]
        a[at] = rng.choice(pool, at.size)
    return t


def assert_same_up_to_nan_payload(devs, ref):
    """Every result that is not NaN bit-identical to the oracle's; NaN exactly
    where the oracle's is NaN (IEEE 754 leaves a NaN result's payload open,
    and the GPU and the host CPUs pick different ones); the bf16 copy of a
    NaN parameter is a bf16 NaN.  Returns the number of NaN parameters."""
    nan_p = 0
    for d, r in zip(devs, ref):
        for k in "pmv":
            a, b = host(d[k], np.uint32), r[k].view(np.uint32)
            bn = np.isnan(r[k])
            assert np.array_equal(np.isnan(a.view(np.float32)), bn), "%s: NaN positions differ" % k
            bad = np.nonzero((a != b) & ~bn)[0]
            assert bad.size == 0, "%s differs at %s: %s vs %s" % (k, bad[:5], a[bad[:5]], b[bad[:5]])
        w, pn = host(d["w"], np.uint16), np.isnan(r["p"])
        assert np.array_equal(w[~pn], r["w"][~pn]), "w differs"
        assert np.all((w[pn] & 0x7FFF) > 0x7F80), "w of a NaN parameter is not a bf16 NaN"
        nan_p += int(pn.sum())
    return nan_p


@pytest.mark.parametrize("step", [1, 18])
def test_non_finite_inputs(step):
    """Infinite and NaN inputs through the fp32 commit: results equal the
    oracle's up to NaN payloads, infinities included.  The digests cannot be
    the oracle's where a NaN was written, so they are checked against the
    verification pass over the written buffers and against a second run."""
    tensors = [nonfinite(40000, step), nonfinite(333, step + 7)]
    runs = []
    for _ in range(2):
        devs, dgot, ref, _ = run_small([dict(t, p=t["p"].copy(), m=t["m"].copy(), v=t["v"].copy())
                                        for t in tensors], step)
        nan_p = assert_same_up_to_nan_payload(devs, ref)
        assert 1000 < nan_p < 40333 - 10000          # both kinds of result are well represented
        assert any(np.isinf(r["p"]).any() for r in ref) and any(np.isinf(r["v"]).any() for r in ref)
        bufs = [b for d, t in zip(devs, tensors) for b in apc.state_buffers(d["p"], d["m"], d["v"], d["w"], t["goff"])]
        assert apc.digests_to_host(apc.digest(bufs, 4)) == dgot
        runs.append((dgot, [host(d[k], np.uint32).copy() for d in devs for k in "pmv"]))
    assert runs[0][0] == runs[1][0]
    assert all(np.array_equal(a, b) for a, b in zip(runs[0][1], runs[1][1]))


def test_commit_zero_grad_reaches_committed_boundary():
    """With APC_COMMIT_ZERO_GRAD the same pass zeroes every gradient: outputs
    and digests equal the oracle's, the guard counts the oracle's nonzero
    gradients before and none after."""
    tensors = [gen(n, off, 5) for n, off in ((50000, 0), (77, 50000), (123457, 50077))]
    want_nz = sum(oracle.count_nonzero(t["g"]) for t in tensors)
    devs, entries = [], []
    for t in tensors:
        d = dict(p=dev(t["p"]), m=dev(t["m"]), v=dev(t["v"]), g=dev(t["g"]),
                 w=torch.zeros(t["p"].size, dtype=torch.int16, device="cuda"))
        devs.append(d)
        entries.append(apc.TensorEntry(d["p"], d["m"], d["v"], d["g"], d["w"], t["goff"]))
    gb = [apc.BufferEntry(d["g"], 0, 0, apc.BF16) for d in devs]
    before = apc.digests_to_host(apc.count_nonzero(gb, 1))
    out = apc.commit_step(entries, 5, HP, zero_grad=True)
    after = apc.digests_to_host(apc.count_nonzero(gb, 1))
    torch.cuda.synchronize()
    assert before == [want_nz] and after == [0]
    h8 = oracle.resolve_hparams(HP, 5)
    ref = [dict(p=t["p"].copy(), m=t["m"].copy(), v=t["v"].copy(), g=t["g"], goff=t["goff"]) for t in tensors]
    ws, dref = oracle.commit_table(ref, h8)
    for r, wv in zip(ref, ws):
        r["w"] = wv
    assert_same(devs, apc.digests_to_host(out), ref, dref)


def test_count_nonzero_of_arbitrary_buffers():
    rng = np.random.default_rng(31)
    bufs, want, keep = [], [0] * 8, []
    for i in range(1100):
        n = int(rng.integers(0, 900))
        slot = int(rng.integers(0, 8))
        f32 = bool(rng.integers(0, 2))
        shift = int(rng.integers(0, 8))
        if f32:
            a = rng.integers(0, 2**32, size=n + shift, dtype=np.uint64).astype(np.uint32)
            a[rng.random(n + shift) < 0.6] = 0
            a[rng.random(n + shift) < 0.05] = 0x80000000
            t = torch.from_numpy(a.view(np.int32)).cuda()
        else:
            a = rng.integers(0, 2**16, size=n + shift, dtype=np.uint64).astype(np.uint16)
            a[rng.random(n + shift) < 0.6] = 0
            a[rng.random(n + shift) < 0.05] = 0x8000
            t = torch.from_numpy(a.view(np.int16)).cuda()
        want[slot] += oracle.count_nonzero(a[shift:])
        keep.append(t)
        bufs.append(apc.BufferEntry(t[shift:], slot, 0, apc.F32 if f32 else apc.BF16))
    assert apc.digests_to_host(apc.count_nonzero(bufs, 8)) == want


def test_count_buffers_at_tile_boundaries():
    """The guard kernel's own tiles: buffers whose bodies end on, just before
    and just after its tile boundaries (and the verification kernel's), with
    and without a scalar head, counted into four slots as numpy counts."""
    rng = np.random.default_rng(34)
    bufs, want, keep = [], [0] * 4, []
    sizes = [k * t + d for t in (COUNT_TILE, DIGEST_TILE) for k in (1, 2) for d in (-8, -1, 0, 1, 9)]
    for i, n in enumerate(sizes):
        for f32 in (True, False):
            shift = int(rng.integers(1, 8)) if i % 2 else 0
            slot = (2 * i + f32) % 4
            dt = np.uint32 if f32 else np.uint16
            a = rng.integers(0, 2 ** (32 if f32 else 16), size=n + shift, dtype=np.uint64).astype(dt)
            a[rng.random(n + shift) < 0.5] = 0
            t = torch.from_numpy(a.view(np.int32 if f32 else np.int16)).cuda()
            want[slot] += oracle.count_nonzero(a[shift:])
            keep.append(t)
            bufs.append(apc.BufferEntry(t[shift:], slot, 0, apc.F32 if f32 else apc.BF16))
    assert apc.digests_to_host(apc.count_nonzero(bufs, 4)) == want


# --------------------------------------------------------- bf16 state (f3)

from apc_testlib import DeviceWorkloadBF16, oracle_at_bf16, oracle_workload_digest_bf16  # noqa: E402


def gen16(n, goff, step):
    p, m, v = synth.state_bf16(n, goff)
    return dict(p=p, m=m, v=v, g=synth.grad(n, goff, step), goff=goff)


def run_bf16(tensors, step, hp=HP, zero_grad=False, shift=0):
    """Commit bf16-state tensors (each optionally viewed `shift` elements
    into its buffers) and compare every word and digest with the oracle."""
    devs, entries = [], []
    for t in tensors:
        n = t["p"].size
        d = {k: dev(np.concatenate([np.zeros(shift, np.uint16), t[k]])) for k in "pmvg"}
        devs.append(d)
        sl = slice(shift, shift + n)
        entries.append(apc.TensorEntryBF16(d["p"][sl], d["m"][sl], d["v"][sl], d["g"][sl], t["goff"]))
    out = apc.commit_step_bf16(entries, step, hp, zero_grad=zero_grad)
    torch.cuda.synchronize()
    h8 = oracle.resolve_hparams(hp, step)
    want = [0, 0, 0]
    for t, d in zip(tensors, devs):
        p, m, v = t["p"].copy(), t["m"].copy(), t["v"].copy()
        dd = oracle.commit_bf16(p, m, v, t["g"], t["goff"], h8)
        want = [(a + b) & M64 for a, b in zip(want, dd)]
        sl = slice(shift, shift + p.size)
        for k, ref in (("p", p), ("m", m), ("v", v)):
            assert np.array_equal(host(d[k], np.uint16)[sl], ref), k
        g_after = host(d["g"], np.uint16)[sl]
        assert (not g_after.any()) if zero_grad else np.array_equal(g_after, t["g"])
    assert apc.digests_to_host(out) == want


def test_bf16_state_non_finite_inputs():
    """Infinite and NaN bf16 words through the bf16-state commit.  Each result
    is the binary32 step rounded once to bf16: where the fp32 oracle's result
    on the widened inputs is NaN the word is a bf16 NaN, elsewhere it equals
    the bf16 oracle's word; the digests equal the verification pass's."""
    rng = np.random.default_rng(52)
    n, step = 30011, 9
    t = gen16(n, 5000, step)
    specials = np.concatenate([np.array([0x7F80, 0xFF80], np.uint16), BF16_NAN])
    for k in "pmvg":
        at = rng.random(n) < 0.04
        t[k][at] = rng.choice(specials, int(at.sum()))
    t["v"][rng.random(n) < 0.02] |= 0x8000                         # negative second moments
    d = {k: dev(t[k]) for k in "pmvg"}
    out = apc.commit_step_bf16([apc.TensorEntryBF16(d["p"], d["m"], d["v"], d["g"], t["goff"])], step, HP)
    got = apc.digests_to_host(out)
    h8 = oracle.resolve_hparams(HP, step)
    p, m, v = t["p"].copy(), t["m"].copy(), t["v"].copy()
    oracle.commit_bf16(p, m, v, t["g"], t["goff"], h8)
    p32, m32, v32 = gf32(t["p"]), gf32(t["m"]), gf32(t["v"])
    oracle.adamw(p32, m32, v32, t["g"], h8)
    for k, ref16, ref32 in (("p", p, p32), ("m", m, m32), ("v", v, v32)):
        a, nan = host(d[k], np.uint16), np.isnan(ref32)
        assert np.array_equal(a[~nan], ref16[~nan]), k
        assert np.all((a[nan] & 0x7FFF) > 0x7F80), k
        assert 0 < nan.sum() < n // 2, k
    assert np.isinf(gf32(p)).any()
    assert apc.digests_to_host(apc.digest(apc.state_buffers_bf16(d["p"], d["m"], d["v"], t["goff"]), 3)) == got


# Elements per tile of the commit kernel's bf16-state layout (27 x 32 threads x 3 groups of 4).
COMMIT_TILE_BF16 = 10368


@pytest.mark.parametrize("n", [1, 3, 7, 8, 9, 63, 4864, 4871, 9728 + 5, 100003] +
                         [k * COMMIT_TILE_BF16 + d for k in (1, 2) for d in (-8, -1, 0, 1, 8)])
def test_bf16_state_sizes(n):
    run_bf16([gen16(n, (1 << 32) - n // 3, 2)], 2)


@pytest.mark.parametrize("shift", [1, 3, 5, 7])
def test_bf16_state_misaligned_views(shift):
    run_bf16([gen16(20000, 77, 3), gen16(513, 20077, 3)], 3, shift=shift)


def test_bf16_state_mutual_misalignment_runs_scalar():
    n = 5000
    t = gen16(n + 8, 0, 4)
    d = {k: dev(t[k]) for k in "pmvg"}
    e = apc.TensorEntryBF16(d["p"][1:n + 1], d["m"][1:n + 1], d["v"][1:n + 1], d["g"][0:n], 9)
    out = apc.commit_step_bf16([e], 4, HP)
    torch.cuda.synchronize()
    p, m, v = t["p"][1:n + 1].copy(), t["m"][1:n + 1].copy(), t["v"][1:n + 1].copy()
    want = oracle.commit_bf16(p, m, v, np.ascontiguousarray(t["g"][0:n]), 9, oracle.resolve_hparams(HP, 4))
    assert np.array_equal(host(d["p"], np.uint16)[1:n + 1], p)
    assert np.array_equal(host(d["v"], np.uint16)[1:n + 1], v)
    assert apc.digests_to_host(out) == want


def test_bf16_state_many_tensors_zero_grad_and_hparams():
    rng = np.random.default_rng(41)
    tensors, off = [], 12345
    for n in rng.integers(1, 2000, size=500):
        tensors.append(gen16(int(n), off, 6))
        off += int(n)
    run_bf16(tensors, 6, zero_grad=True)
    run_bf16(tensors[:40], 1000, dict(lr=1e-2, beta1=0.0, beta2=0.999, eps=1e-6, weight_decay=0.0))


def test_f3_rank_shard_bf16_full_size():
    """The paper's 4-way rank shard of Mistral-7B in bf16 state (1,812,005,888
    elements, 77 pieces of one allocation): sampled words against the
    oracle, the verification digest equals the fused one, and the digests of
    a 64 Mi-element slice equal the streamed oracle's."""
    w = W.f3()
    dw = DeviceWorkloadBF16(w, 5)
    got = apc.digests_to_host(apc.commit_step_bf16(dw.entries(), 5, HP))
    idx = sample_indices(w, 200000, 7)
    res = dw.gather(idx)
    ref = oracle_at_bf16(idx, 5)
    for k in "pmv":
        assert np.array_equal(res[k], ref[k]), k
    assert apc.digests_to_host(apc.digest(dw.digest_buffers(), 3)) == got
    lo = w.pieces[0].goff + 123_456_789
    hi = lo + (64 << 20)
    start = lo - (w.pieces[0].goff - w.pieces[0].at)
    b = dw.bufs[0]
    sl = slice(start, start + (hi - lo))
    part = apc.digests_to_host(apc.digest(apc.state_buffers_bf16(b["p"][sl], b["m"][sl], b["v"][sl], lo), 3))
    assert part == oracle_workload_digest_bf16(w, 5, lo, hi)
    del dw
    torch.cuda.empty_cache()


def test_single_entry_longer_than_2_32_elements():
    """One entry of 2^32 + 4099 elements (64-bit tile and element indices
    inside one tensor, ~69 GB of state): sampled elements against the
    oracle; the same data given as three pieces digests identically; a
    window around the entry's 2^32nd element matches the streamed oracle."""
    free, _ = torch.cuda.mem_get_info()
    if free < 80 * (1 << 30):
        pytest.skip("needs ~75 GB of free device memory")
    n = (1 << 32) + 4099
    goff = 1000
    w1 = W.Workload("big", [W.Piece("flat", n, goff, 0, 0)], [3], chained=False, allocs=[n])
    dw = DeviceWorkload(w1, 3)
    # as three pieces first (ragged cuts), then the state is regenerated and run as one entry
    cuts = [0, 123_456_789, (1 << 32) - 5, n]
    b = dw.bufs[0]
    pieces = [apc.TensorEntry(b["p"][a:c], b["m"][a:c], b["v"][a:c], b["g"][a:c], b["w"][a:c], goff + a)
              for a, c in zip(cuts[:-1], cuts[1:])]
    d3 = apc.digests_to_host(apc.commit_step(pieces, 3, HP))
    dw.fill_state()
    d1 = apc.digests_to_host(apc.commit_step(dw.entries(), 3, HP))
    assert d1 == d3
    idx = np.unique(np.concatenate([sample_indices(w1, 50000, 11),
                                    np.array([goff + (1 << 32) + j for j in (-2, -1, 0, 1, 4098)], dtype=np.uint64)]))
    got = dw.gather(idx)
    ref = oracle_at(idx, 3)
    for key in "pmvw":
        assert np.array_equal(got[key], ref[key]), key
    lo = (1 << 32) - (1 << 20)            # element offsets inside the entry
    hi = (1 << 32) + 4099
    sl = slice(lo, hi)
    part = apc.digests_to_host(apc.digest(apc.state_buffers(b["p"][sl], b["m"][sl], b["v"][sl], b["w"][sl],
                                                            goff + lo), 4))
    wpart = W.Workload("win", [W.Piece("win", hi - lo, goff + lo, 0, 0)], [3], chained=False, allocs=[hi - lo])
    assert part == oracle_workload_digest(wpart, 3)
    del dw, b, pieces
    torch.cuda.empty_cache()


def test_step_captured_in_a_cuda_graph_replays_bit_exact():
    """The step enqueues only a memset and kernel launches on the caller's
    stream, so it can be captured once and replayed; each replay equals the
    eager path step for step (chained state) and the oracle."""
    tensors = [gen(n, off, 4) for n, off in ((70000, 0), (5, 70000), (33333, 70005))]
    devs, entries = [], []
    for t in tensors:
        d = dict(p=dev(t["p"]), m=dev(t["m"]), v=dev(t["v"]), g=dev(t["g"]),
                 w=torch.zeros(t["p"].size, dtype=torch.int16, device="cuda"))
        devs.append(d)
        entries.append(apc.TensorEntry(d["p"], d["m"], d["v"], d["g"], d["w"], t["goff"]))
    vb = [b for e in entries for b in apc.state_buffers(e.p, e.m, e.v, e.w, e.global_offset)]
    out_c = torch.empty(4, dtype=torch.int64, device="cuda")
    out_v = torch.empty(4, dtype=torch.int64, device="cuda")
    apc.commit_step(entries, 4, HP, out=out_c)        # first call: per-device queries happen outside capture
    torch.cuda.synchronize()
    for t, d in zip(tensors, devs):                   # back to the generated state
        for k in "pmv":
            d[k].copy_(torch.from_numpy(t[k]).cuda())
    s = torch.cuda.Stream()
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.stream(s):
        with torch.cuda.graph(graph, stream=s):
            apc.commit_step(entries, 4, HP, stream=s, out=out_c)
            apc.digest(vb, 4, stream=s, out=out_v)
    torch.cuda.synchronize()
    for t, d in zip(tensors, devs):                   # capture does not run the work: reset anyway
        for k in "pmv":
            d[k].copy_(torch.from_numpy(t[k]).cuda())
    h8 = oracle.resolve_hparams(HP, 4)
    ref = [dict(p=t["p"].copy(), m=t["m"].copy(), v=t["v"].copy(), g=t["g"], goff=t["goff"]) for t in tensors]
    for rep in range(3):                              # three chained steps, all with t = 4
        graph.replay()
        torch.cuda.synchronize()
        ws, dref = oracle.commit_table(ref, h8)
        for r, wv in zip(ref, ws):
            r["w"] = wv
        assert_same(devs, apc.digests_to_host(out_c), ref, dref)
        assert apc.digests_to_host(out_v) == dref


def test_concurrent_host_threads_on_separate_streams():
    """Four host threads, each with its own stream and tables, call the
    step and the digest repeatedly at the same time; every result equals
    the oracle's (the library's per-device state and per-thread error
    state are shared safely)."""
    import threading
    jobs = []
    for j in range(4):
        tensors = [gen(n, off, 2) for n, off in ((20_000 + 17 * j, (1 << 32) - 7_000 * (j + 1)), (9, 10 ** 6 * (j + 1)))]
        devs = [dict(p=dev(t["p"]), m=dev(t["m"]), v=dev(t["v"]), g=dev(t["g"]),
                     w=torch.zeros(t["p"].size, dtype=torch.int16, device="cuda")) for t in tensors]
        jobs.append((tensors, devs))
    torch.cuda.synchronize()
    results, errors = [None] * 4, []

    def work(j):
        try:
            tensors, devs = jobs[j]
            s = torch.cuda.Stream()
            entries = [apc.TensorEntry(d["p"], d["m"], d["v"], d["g"], d["w"], t["goff"]) for d, t in zip(devs, tensors)]
            vb = [b for e in entries for b in apc.state_buffers(e.p, e.m, e.v, e.w, e.global_offset)]
            got = []
            for _ in range(5):                        # five chained steps, t = 2
                with torch.cuda.stream(s):
                    oc = apc.commit_step(entries, 2, HP, stream=s)
                    ov = apc.digest(vb, 4, stream=s)
                s.synchronize()
                got.append((apc.digests_to_host(oc), apc.digests_to_host(ov)))
            results[j] = got
        except Exception as e:  # reported by the main thread
            errors.append(repr(e))

    threads = [threading.Thread(target=work, args=(j,)) for j in range(4)]
    for t in threads:
        t.start()
    for t in threads:
        t.join()
    assert not errors, errors
    h8 = oracle.resolve_hparams(HP, 2)
    for j, (tensors, devs) in enumerate(jobs):
        ref = [dict(p=t["p"].copy(), m=t["m"].copy(), v=t["v"].copy(), g=t["g"], goff=t["goff"]) for t in tensors]
        for k in range(5):
            ws, dref = oracle.commit_table(ref, h8)
            for r, wv in zip(ref, ws):
                r["w"] = wv
            assert results[j][k] == (dref, dref), (j, k)
        assert_same(devs, dref, ref, dref)


@pytest.mark.parametrize("value", ["", "abc", "0", "-5", "12x", "99999999999999999999"])
def test_malformed_grid_limit_is_ignored(monkeypatch, value):
    monkeypatch.setenv("APC_GRID_LIMIT", value)
    tensors = [gen(n, off, 3) for n, off in ((50_001, 123), (6, 50_124))]
    assert_same(*run_small(tensors, 3))


def test_bf16_copy_of_every_binary32_pattern():
    """With lr = 0 and m = v = g = 0 the step leaves p' = p exactly, so w is
    the kernel's bf16 rounding of p itself.  Every one of the 2^32 bit
    patterns goes through the commit kernel in chunks of 2^28: p' and w
    equal the oracle's bit for bit (NaNs excepted: outside the contract),
    and the fused digests of p', m', v', w equal the oracle's (chunks with
    NaNs excepted), which pins the commit kernel's own splitmix64 form on
    every low word."""
    from concurrent.futures import ThreadPoolExecutor
    hp = dict(HP, lr=0.0)
    chunk = 1 << 28
    p = torch.empty(chunk, dtype=torch.int32, device="cuda")
    m = torch.zeros(chunk, dtype=torch.float32, device="cuda")
    v = torch.zeros(chunk, dtype=torch.float32, device="cuda")
    g = torch.zeros(chunk, dtype=torch.int16, device="cuda")
    w = torch.empty(chunk, dtype=torch.int16, device="cuda")
    out = torch.empty(4, dtype=torch.int64, device="cuda")
    tab = apc.prepare_table([apc.TensorEntry(p, m, v, g, w, 0)])
    base = np.arange(chunk, dtype=np.uint32)
    u = np.empty_like(base)
    zero_digest = oracle.digest_f32(np.zeros(chunk, dtype=np.uint32), 0)

    def expected(start):
        a = base + np.uint32(start)
        return oracle.digest_f32(a, 0), oracle.digest_u16(oracle.bf16_rne(a.view(np.float32)), 0)

    pool = ThreadPoolExecutor(4)
    pending = []
    for start in range(0, 1 << 32, chunk):
        p.copy_(torch.arange(start, start + chunk, dtype=torch.int64, device="cuda").to(torch.int32))
        m.zero_()
        v.zero_()
        d = apc.digests_to_host(apc.commit_step(tab, 1, hp, out=out))
        np.add(base, np.uint32(start), out=u)
        f = u.view(np.float32)
        keep = ~np.isnan(f)
        got_p = p.cpu().numpy().view(np.uint32)
        got_w = w.cpu().numpy().view(np.uint16)
        assert np.array_equal(got_p[keep], u[keep]), hex(start)
        assert np.array_equal(got_w[keep], oracle.bf16_rne(f)[keep]), hex(start)
        assert d[1] == zero_digest and d[2] == zero_digest, hex(start)
        if keep.all():
            pending.append((start, d, pool.submit(expected, start)))
    for start, d, fut in pending:
        dp, dw = fut.result()
        assert d[0] == dp and d[3] == dw, hex(start)
    pool.shutdown()
    assert len(pending) == 14                     # the two chunks holding NaN patterns are left out
    del p, m, v, g, w
    torch.cuda.empty_cache()


def test_digest_of_every_low_word():
    """A buffer whose element i holds bits i (i < 2^32), digested at global
    offset 0 in chunks of 2^28: the keys (i << 32) | i cover every low word
    and every index mod 2^32 once.  The wrapping sum of the GPU's chunk
    digests equals the oracle's (digest concatenation)."""
    from concurrent.futures import ThreadPoolExecutor
    chunk = 1 << 28
    starts = list(range(0, 1 << 32, chunk))
    buf = torch.empty(chunk, dtype=torch.int32, device="cuda")
    out = torch.empty(1, dtype=torch.int64, device="cuda")
    got = 0
    for start in starts:
        buf.copy_(torch.arange(start, start + chunk, dtype=torch.int64, device="cuda").to(torch.int32))
        got = (got + apc.digests_to_host(apc.digest([apc.BufferEntry(buf, 0, start, apc.F32)], 1, out=out))[0]) & M64

    def part(start):
        return oracle.digest_f32(np.arange(chunk, dtype=np.uint32) + np.uint32(start), start)

    with ThreadPoolExecutor(4) as ex:
        want = sum(ex.map(part, starts)) & M64
    assert got == want
    del buf
    torch.cuda.empty_cache()


def test_every_bf16_parameter_and_gradient_pair():
    """Every pair (p, g) of a bf16 bit pattern p (widened to binary32) and a
    bf16 gradient g, 2^32 elements at m = v = 0, through the fp32 commit
    kernel in chunks of 2^28; NaN parameters and non-finite gradients, which
    are outside the contract, are replaced by +0.  p', m', v', w and the
    four digests equal the oracle's bit for bit."""
    import os
    chunk = 1 << 28
    nthreads = os.cpu_count() or 1
    step = 3
    h8 = oracle.resolve_hparams(HP, step)
    idx = np.arange(chunk, dtype=np.uint32)
    d = {k: torch.empty(chunk, dtype=torch.float32, device="cuda") for k in "pmv"}
    d["g"] = torch.empty(chunk, dtype=torch.int16, device="cuda")
    d["w"] = torch.empty(chunk, dtype=torch.int16, device="cuda")
    out = torch.empty(4, dtype=torch.int64, device="cuda")
    tab = apc.prepare_table([apc.TensorEntry(d["p"], d["m"], d["v"], d["g"], d["w"], 0)])
    for start in range(0, 1 << 32, chunk):
        i = idx + np.uint32(start)
        p16 = (i >> 16).astype(np.uint16)
        g16 = (i & 0xFFFF).astype(np.uint16)
        p16[(p16 & 0x7FFF) > 0x7F80] = 0                     # NaN parameters
        g16[(g16 & 0x7FFF) >= 0x7F80] = 0                    # infinite and NaN gradients
        p = (p16.astype(np.uint32) << 16).view(np.float32)
        m = np.zeros(chunk, dtype=np.float32)
        v = np.zeros(chunk, dtype=np.float32)
        d["p"].copy_(torch.from_numpy(p))
        d["m"].zero_()
        d["v"].zero_()
        d["g"].copy_(torch.from_numpy(g16.view(np.int16)))
        got = apc.digests_to_host(apc.commit_step(tab, step, HP, out=out))
        w, dref = oracle.commit(p, m, v, g16, 0, h8, nthreads=nthreads)
        for k, ref in (("p", p), ("m", m), ("v", v)):
            a = d[k].cpu().numpy().view(np.uint32)
            bad = np.nonzero(a != ref.view(np.uint32))[0]
            assert bad.size == 0, (hex(start), k, bad[:4])
        assert np.array_equal(d["w"].cpu().numpy().view(np.uint16), w), hex(start)
        assert got == dref, hex(start)
    del d
    torch.cuda.empty_cache()


def test_every_bf16_state_parameter_and_gradient_pair():
    """The bf16-state step (the paper's precision) over every pair (p, g) of
    bf16 bit patterns, 2^32 elements at m = v = 0, in chunks of 2^28; NaN
    parameters and non-finite gradients are replaced by +0.  p', m', v' and
    the three digests equal the oracle's bit for bit."""
    import os
    from concurrent.futures import ThreadPoolExecutor
    chunk, sub = 1 << 28, 1 << 24
    step = 3
    h8 = oracle.resolve_hparams(HP, step)
    idx = np.arange(chunk, dtype=np.uint32)
    d = {k: torch.empty(chunk, dtype=torch.int16, device="cuda") for k in "pmvg"}
    out = torch.empty(3, dtype=torch.int64, device="cuda")
    tab = apc.prepare_table([apc.TensorEntryBF16(d["p"], d["m"], d["v"], d["g"], 0)])
    pool = ThreadPoolExecutor(os.cpu_count() or 1)
    for start in range(0, 1 << 32, chunk):
        i = idx + np.uint32(start)
        p = (i >> 16).astype(np.uint16)
        g = (i & 0xFFFF).astype(np.uint16)
        p[(p & 0x7FFF) > 0x7F80] = 0                          # NaN parameters
        g[(g & 0x7FFF) >= 0x7F80] = 0                         # infinite and NaN gradients
        m = np.zeros(chunk, dtype=np.uint16)
        v = np.zeros(chunk, dtype=np.uint16)
        d["p"].copy_(torch.from_numpy(p.view(np.int16)))
        d["m"].zero_()
        d["v"].zero_()
        d["g"].copy_(torch.from_numpy(g.view(np.int16)))
        got = apc.digests_to_host(apc.commit_step_bf16(tab, step, HP, out=out))
        parts = pool.map(lambda s: oracle.commit_bf16(p[s:s + sub], m[s:s + sub], v[s:s + sub], g[s:s + sub], s, h8),
                         range(0, chunk, sub))
        want = [0, 0, 0]
        for dd in parts:
            want = [(a + b) & M64 for a, b in zip(want, dd)]
        for k, ref in (("p", p), ("m", m), ("v", v)):
            a = d[k].cpu().numpy().view(np.uint16)
            bad = np.nonzero(a != ref)[0]
            assert bad.size == 0, (hex(start), k, bad[:4])
        assert got == want, hex(start)
    pool.shutdown()
    del d
    torch.cuda.empty_cache()


@pytest.mark.parametrize("k", [0, 1, 2, 3])
def test_groups_straddling_a_top_bits_boundary(k):
    """The commit kernel shares hi >> 30 of the incremented key high word
    (G + 0x9E3779B9 + carry) across a group of four elements unless the
    group's range crosses a multiple of 2^30.  Tensors around each of the
    four crossing points take both the shared and the exact path; outputs
    and digests equal the oracle's."""
    cross = ((k << 30) - 0x9E3779B9) & 0xFFFFFFFF      # the key index G at which the top bits change
    tensors = [gen(n, cross - back + (1 << 32) * j, 2) for j, (n, back) in enumerate(((20_000, 9_999), (13, 7), (4_867, 4_800)))]
    assert_same(*run_small(tensors, 2))


@pytest.mark.parametrize("k", [0, 1, 2, 3])
def test_verify_tiles_straddling_a_top_bits_boundary(k):
    """The verification pass shares hi >> 30 across a thread's terms in a
    tile unless their keys' range crosses a multiple of 2^30 after the
    increment; buffers around each crossing point (fp32 and bf16, aligned
    and not) digest as the oracle does."""
    rng = np.random.default_rng(40 + k)
    cross = ((k << 30) - 0x9E3779B9) & 0xFFFFFFFF
    bufs, want, keep = [], [0, 0], []
    for back, n, shift in ((60_000, 120_001, 0), (7, 20, 1), (12_300, 30_000, 3)):
        goff = cross - back + (1 << 33)
        a = rng.integers(0, 2**32, size=n + shift, dtype=np.uint64).astype(np.uint32)
        t = torch.from_numpy(a.view(np.int32)).cuda()
        keep.append(t)
        bufs.append(apc.BufferEntry(t[shift:], 0, goff, apc.F32))
        want[0] = (want[0] + oracle.digest_f32(a[shift:], goff)) & M64
        h = rng.integers(0, 2**16, size=n + shift, dtype=np.uint64).astype(np.uint16)
        th = torch.from_numpy(h.view(np.int16)).cuda()
        keep.append(th)
        bufs.append(apc.BufferEntry(th[shift:], 1, goff, apc.BF16))
        want[1] = (want[1] + oracle.digest_u16(h[shift:], goff)) & M64
    assert apc.digests_to_host(apc.digest(bufs, 2)) == want


def test_every_bf16_word_digested_at_every_crossing():
    """Every 16-bit word, digested by the verification pass (fp32 words are
    covered by test_digest_of_every_low_word) at offsets that put the
    shared-top-bits check on both sides of each 2^30 crossing, equals the
    oracle's digest."""
    words = np.arange(1 << 16, dtype=np.uint32).astype(np.uint16)
    t = torch.from_numpy(words.view(np.int16)).cuda()
    bufs, want = [], [0]
    for k in range(4):
        cross = ((k << 30) - 0x9E3779B9) & 0xFFFFFFFF
        for j, back in enumerate((0, 1, 4_000, 60_000, 65_535)):
            goff = cross - back + (j << 32)
            bufs.append(apc.BufferEntry(t, 0, goff, apc.BF16))
            want[0] = (want[0] + oracle.digest_u16(words, goff)) & M64
    assert apc.digests_to_host(apc.digest(bufs, 1)) == want
