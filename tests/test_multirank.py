"""The multi-rank path on CPU ranks (Gloo, world size 2): each rank commits
its own shard (here with the oracle standing in for the device), the ranks
bracket the step with barriers and a max-over-ranks time, then exchange their
32-byte digests on the control plane.  The whole-model digest is the wrapping
sum of the shard digests (concatenation), and a bit flipped on one rank's
host copy before its verification is caught by every rank (fail-stop on a
failed validation, the paper's Section III-C safety invariant)."""
import multiprocessing as mp
import os
import socket

import numpy as np
import pytest

SIZES = [3000, 1, 4099]            # one rank's table: ragged tensors
PER_RANK = sum(SIZES)
STEP = 4


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _model(world):
    """A small flat model: the rank tables of the copy partition, laid end
    to end, as one workload to cut with the model partition."""
    from synth import workloads as W
    pieces, off = [], 0
    for r in range(world):
        for n in SIZES:
            pieces.append(W.Piece("t%d" % len(pieces), n, off, alloc=len(pieces)))
            off += n
    return W.Workload("small", pieces, [STEP], False, allocs=[pc.n for pc in pieces])


def _rank_main(rank, world, port, flip_rank, q, split="copy"):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(world),
                      LOCAL_RANK=str(rank))
    try:
        import bench
        import oracle
        import synth
        from synth import workloads as W
        dist = bench.init_control_plane(world)
        if split == "model":    # rank r: the contiguous range r of the one model (bench --split model)
            pieces = [(pc.n, pc.goff) for pc in W.shard(_model(world), rank, world).pieces]
        else:                   # rank r: a full-size copy at offset r * N (bench --split copy)
            base = bench.shard_offset(rank, PER_RANK)
            pieces = [(n, base + sum(SIZES[:k])) for k, n in enumerate(SIZES)]
        h8 = oracle.resolve_hparams(oracle.DEFAULT_HP, STEP)
        bench.barrier(dist)
        commit, verify = [0, 0, 0, 0], [0, 0, 0, 0]
        for k, (n, off) in enumerate(pieces):
            p, m, v = synth.state(n, off, nthreads=1)
            g = synth.grad(n, off, STEP, nthreads=1)
            w, d = oracle.commit(p, m, v, g, off, h8)
            commit = [(a + b) & bench.M64 for a, b in zip(commit, d)]
            if rank == flip_rank and k == 0:
                p.view(np.uint32)[17] ^= np.uint32(1 << 9)      # host-side fault injection
            dv = [oracle.digest_f32(p, off), oracle.digest_f32(m, off), oracle.digest_f32(v, off),
                  oracle.digest_u16(w, off)]
            verify = [(a + b) & bench.M64 for a, b in zip(verify, dv)]
        t = bench.max_over_ranks(dist, float(rank + 1))
        summed = bench.sum_over_ranks(dist, commit)
        bench.barrier(dist)
        from paper_2609_18178_gb300 import cohort
        try:
            whole, verified = bench.exchange_digests(dist, STEP, commit, verify, shard=rank)
            outcome = "agreed"
        except cohort.CohortMismatch as e:
            whole, verified, outcome = None, False, "mismatch:%s:%s" % (e.what, e.ranks)
        dist.destroy_process_group()
        q.put((rank, t, whole, verified, outcome, summed))
    except Exception as e:  # report to the parent instead of hanging it
        q.put((rank, "error", repr(e), None, None))


def _run(world, flip_rank, split="copy"):
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_rank_main, args=(r, world, port, flip_rank, q, split)) for r in range(world)]
    for p in procs:
        p.start()
    res = [q.get(timeout=240) for _ in procs]
    for p in procs:
        p.join(timeout=60)
    assert all(r[1] != "error" for r in res), res
    return sorted(res)


def _whole_model_digest(world):
    import oracle
    import synth
    h8 = oracle.resolve_hparams(oracle.DEFAULT_HP, STEP)
    tot, off = [0, 0, 0, 0], 0
    for _ in range(world):
        for n in SIZES:
            p, m, v = synth.state(n, off, nthreads=1)
            g = synth.grad(n, off, STEP, nthreads=1)
            _, d = oracle.commit(p, m, v, g, off, h8)
            tot = [(a + b) % (1 << 64) for a, b in zip(tot, d)]
            off += n
    return tot


@pytest.mark.parametrize("split", ["copy", "model"])
def test_two_ranks_exchange_digests(split):
    """Both partitions of bench.py: full-size copies at offsets r * N, or
    the contiguous halves of one flat model of the same 2N elements; either
    way the ranks' digests add up to the whole model's."""
    res = _run(2, flip_rank=-1, split=split)
    want = _whole_model_digest(2)
    for rank, t, whole, verified, outcome, summed in res:
        assert t == 2.0                      # max over ranks of (rank + 1)
        assert outcome == "agreed" and verified
        assert whole == want                 # concatenation: shards sum to the whole model
        assert summed == want                # the all-reduce of the first-step digests
    assert res[0][2] == res[1][2]


def test_host_fault_on_one_rank_is_seen_by_all():
    res = _run(2, flip_rank=1)
    for rank, t, whole, verified, outcome, summed in res:
        assert outcome == "mismatch:verification:[1]"
