"""Cohort agreement on the committed state, over the host control plane.

After a communicator fault at a committed optimizer boundary, the paper's
recovery protocol (arxiv 2609.18178, Section III-C) has every rank
synchronise on an out-of-band Gloo channel, agree exactly on the committed
frontier F and the generation counter g (phase 3), and validate readiness
before release (phase 6); any error or timeout in those phases makes a
rank stop, and the channel makes the surviving peers stop within a bounded
deadline (the safety invariant).  The ranks of one replication group hold
identical shards (hybrid sharding, Section II-A), and the paper's result is
that those shards stay bit-identical through repairs (Section IV-F).

``agree`` is that exchange with the 32-byte state digests of
``apc_commit_step`` / ``apc_digest`` standing in for the bitwise state
checks: one all-gather of (F, g, guard result, shard id, digests) per rank,
then, on every rank, the same checks:

* every rank reports the same F and the same g           (phase 3)
* every rank's quiescence guard passed                    (phase 2 result)
* every rank's verification pass reproduced its digests  (phase 6)
* all replicas of a shard report identical digests       (phase 6)

The whole-model digest is the wrapping sum of one replica's digests per
shard (the digest is additive over disjoint index ranges).  A failed check
raises ``CohortMismatch`` on every rank; a peer that does not take part
within the process group's timeout makes the collective raise, reported as
``CohortLost``.  Callers stop (fail-stop) on either.

Only host-side logic: it uses torch.distributed with the Gloo backend.
"""
from __future__ import annotations

import time
from dataclasses import dataclass

M64 = (1 << 64) - 1


class CohortError(RuntimeError):
    """The cohort cannot agree: the caller must stop (fail-stop)."""


class CohortMismatch(CohortError):
    """Every rank took part but a check failed."""

    def __init__(self, what: str, ranks: list[int], detail: str = ""):
        super().__init__("cohort disagrees on %s (ranks %s)%s" % (what, ranks, (": " + detail) if detail else ""))
        self.what = what
        self.ranks = ranks


class CohortLost(CohortError):
    """A peer did not take part within the deadline."""


@dataclass
class Report:
    rank: int
    frontier: int
    generation: int
    guard_ok: bool
    verified: bool
    shard: int
    digests: list[int]


@dataclass
class Agreement:
    frontier: int
    generation: int
    whole_digests: list[int]           # wrapping sum over shards
    shard_digests: dict[int, list[int]]
    reports: list[Report]
    seconds: float


def check(reports: list[Report]) -> Agreement:
    """The checks every rank runs on the gathered reports (pure function)."""
    t0 = time.perf_counter()
    fr = {r.frontier for r in reports}
    if len(fr) != 1:
        f0 = reports[0].frontier
        raise CohortMismatch("frontier F", [r.rank for r in reports if r.frontier != f0], "values %s" % sorted(fr))
    gen = {r.generation for r in reports}
    if len(gen) != 1:
        g0 = reports[0].generation
        raise CohortMismatch("generation g", [r.rank for r in reports if r.generation != g0],
                             "values %s" % sorted(gen))
    bad = [r.rank for r in reports if not r.guard_ok]
    if bad:
        raise CohortMismatch("quiescence guard", bad, "outstanding gradients or busy modules")
    bad = [r.rank for r in reports if not r.verified]
    if bad:
        raise CohortMismatch("verification", bad, "the verify pass did not reproduce the commit digests")
    by_shard: dict[int, list[Report]] = {}
    for r in reports:
        by_shard.setdefault(r.shard, []).append(r)
    shard_digests = {}
    for sid, rs in sorted(by_shard.items()):
        ref = [d & M64 for d in rs[0].digests]
        off = [r.rank for r in rs if [d & M64 for d in r.digests] != ref]
        if off:
            raise CohortMismatch("state digests of shard %d" % sid, [rs[0].rank] + off,
                                 "replicas differ bitwise")
        shard_digests[sid] = ref
    width = len(next(iter(shard_digests.values())))
    whole = [0] * width
    for ds in shard_digests.values():
        whole = [(a + b) & M64 for a, b in zip(whole, ds)]
    return Agreement(reports[0].frontier, reports[0].generation, whole, shard_digests, reports,
                     time.perf_counter() - t0)


def agree(dist, frontier: int, generation: int, digests: list[int], shard: int, guard_ok: bool = True,
          verified: bool = True, group=None) -> Agreement:
    """Exchange this rank's report with the cohort and run the checks.

    dist: ``torch.distributed`` with an initialised Gloo process group whose
    timeout is the protocol's deadline.  Raises CohortMismatch or CohortLost
    on every rank; returns the Agreement otherwise."""
    t0 = time.perf_counter()
    me = Report(dist.get_rank(group) if group is not None else dist.get_rank(), int(frontier), int(generation),
                bool(guard_ok), bool(verified), int(shard), [int(d) & M64 for d in digests])
    world = dist.get_world_size(group) if group is not None else dist.get_world_size()
    gathered = [None] * world
    try:
        dist.all_gather_object(gathered, me, group=group)
    except Exception as e:  # a lost or hung peer ends the collective at the deadline
        raise CohortLost("control-plane exchange failed: %s" % (str(e).splitlines()[0] if str(e) else type(e).__name__))
    result = check(gathered)
    result.seconds = time.perf_counter() - t0
    return result
