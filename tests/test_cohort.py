"""Cohort agreement (paper_2609_18178_gb300.cohort) on CPU ranks over Gloo:
the paper's phase-3 frontier agreement, phase-6 validation and fail-stop
safety invariant (Section III-C), with the 32-byte state digests of the
committed step standing in for the bitwise state checks.  Four ranks form
two shards x two replicas (hybrid sharding's replication groups); every
fault is injected on the host: a skewed frontier, a bit flipped in one
replica's state, a failed guard, a peer that leaves before the exchange."""
import datetime
import multiprocessing as mp
import os
import socket
import time

import numpy as np
import pytest

from paper_2609_18178_gb300 import cohort

STEP = 9
SIZES = [2000, 3, 1025]


def _port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def shard_digests(shard, flip=False):
    import oracle
    import synth
    h8 = oracle.resolve_hparams(oracle.DEFAULT_HP, STEP)
    tot, off = [0, 0, 0, 0], shard * sum(SIZES)
    for n in SIZES:
        p, m, v = synth.state(n, off, nthreads=1)
        g = synth.grad(n, off, STEP, nthreads=1)
        w, _ = oracle.commit(p, m, v, g, off, h8)
        if flip and n == SIZES[0]:
            m.view(np.uint32)[5] ^= np.uint32(1 << 20)      # host-side fault injection
        d = [oracle.digest_f32(p, off), oracle.digest_f32(m, off), oracle.digest_f32(v, off),
             oracle.digest_u16(w, off)]
        tot = [(a + b) % (1 << 64) for a, b in zip(tot, d)]
        off += n
    return tot


ROUNDS = [None, "frontier", "flip", "guard"]


def _one_round(dist, grp, rank, fault):
    shard = rank // 2
    frontier = STEP + (1 if fault == "frontier" and rank == 2 else 0)
    guard = not (fault == "guard" and rank == 1)
    d = shard_digests(shard, flip=(fault == "flip" and rank == 3))
    t0 = time.perf_counter()
    try:
        ag = cohort.agree(dist, frontier, 1, d, shard, guard_ok=guard, group=grp)
        return ("agreed", ag.whole_digests, ag.seconds)
    except cohort.CohortMismatch as e:
        return ("mismatch", (e.what, e.ranks), time.perf_counter() - t0)
    except cohort.CohortLost as e:
        return ("lost", str(e)[:80], time.perf_counter() - t0)


def _rank(rank, world, port, rounds, q):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    try:
        import torch.distributed as dist
        # a generous rendezvous (cold imports), then the protocol's own group
        # whose timeout is its 6 s deadline
        dist.init_process_group("gloo", rank=rank, world_size=world, timeout=datetime.timedelta(seconds=120))
        grp = dist.new_group(ranks=list(range(world)), backend="gloo", timeout=datetime.timedelta(seconds=6))
        outcomes = []
        for fault in rounds:
            if fault == "lost" and rank == 3:
                q.put((rank, [("left", None, 0.0)]))
                q.close()
                q.join_thread()                              # flush before leaving
                os._exit(0)                                  # leaves without taking part
            # a mismatch reaches every rank after the exchange, so the group stays usable
            outcomes.append(_one_round(dist, grp, rank, fault))
        q.put((rank, outcomes))
        try:
            dist.destroy_process_group()
        except Exception:
            pass
    except Exception as e:
        q.put((rank, [("error", repr(e), 0.0)]))


def run(rounds, world=4):
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _port()
    ps = [ctx.Process(target=_rank, args=(r, world, port, rounds, q)) for r in range(world)]
    for p in ps:
        p.start()
    out = sorted(q.get(timeout=180) for _ in ps)
    for p in ps:
        p.join(timeout=60)
        if p.is_alive():
            p.kill()
    assert all(o[0] != "error" for r in out for o in r[1]), out
    return out


def test_check_is_a_pure_function_of_the_reports():
    R = cohort.Report
    a, b = [1, 2, 3, 4], [5, 6, 7, 8]
    ag = cohort.check([R(0, 3, 1, True, True, 0, a), R(1, 3, 1, True, True, 0, a), R(2, 3, 1, True, True, 1, b)])
    assert ag.whole_digests == [6, 8, 10, 12] and ag.shard_digests == {0: a, 1: b}
    with pytest.raises(cohort.CohortMismatch) as e:
        cohort.check([R(0, 3, 1, True, True, 0, a), R(1, 4, 1, True, True, 0, a)])
    assert e.value.what == "frontier F" and e.value.ranks == [1]
    with pytest.raises(cohort.CohortMismatch) as e:
        cohort.check([R(0, 3, 1, True, True, 0, a), R(1, 3, 2, True, True, 0, a)])
    assert e.value.what == "generation g"
    with pytest.raises(cohort.CohortMismatch) as e:
        cohort.check([R(0, 3, 1, True, True, 0, a), R(1, 3, 1, True, True, 0, b)])
    assert e.value.what == "state digests of shard 0" and e.value.ranks == [0, 1]
    with pytest.raises(cohort.CohortMismatch) as e:
        cohort.check([R(0, 3, 1, True, False, 0, a)])
    assert e.value.what == "verification"
    m = (1 << 64) - 1
    assert cohort.check([R(0, 1, 1, True, True, 0, [m] * 4), R(1, 1, 1, True, True, 1, [2] * 4)]).whole_digests == [1] * 4


def test_four_ranks_agree_then_every_fault_stops_every_rank():
    """Rounds on one process group: agreement, then a skewed frontier, a bit
    flipped in one replica's state and a failed guard, each reported to
    every rank."""
    out = run(ROUNDS)
    want = [(a + b) % (1 << 64) for a, b in zip(shard_digests(0), shard_digests(1))]
    for rank, outcomes in out:
        ok, frontier, flip, guard = outcomes
        assert ok[0] == "agreed" and ok[1] == want        # shards sum to the whole model
        assert frontier[:2] == ("mismatch", ("frontier F", [2]))
        assert flip[:2] == ("mismatch", ("state digests of shard 1", [2, 3]))
        assert guard[:2] == ("mismatch", ("quiescence guard", [1]))
    print("cohort agreement, 4 CPU ranks over Gloo on one host: %.2f ms max"
          % (1e3 * max(o[1][0][2] for o in out)))


def test_lost_peer_stops_the_others_within_the_deadline():
    out = run([None, "lost"])
    assert out[3][1] == [("left", None, 0.0)]
    for rank, outcomes in out[:3]:
        assert outcomes[0][0] == "agreed"
        kind, detail, secs = outcomes[1]
        assert kind == "lost", (rank, kind, detail)
        assert secs < 6.0 + 10.0          # the process group's 6 s deadline, plus slack
