"""Tensor tables of the committed-step workloads (shapes, offsets, steps).

Shapes follow the paper's models (arxiv 2609.18178, Section IV-A):
Mistral-7B-v0.3 with 7,248,023,552 parameters (Table III caption and the
macro workload text), sharded 4-way intra-node x 4-way inter-node on 16 GPUs,
and the 1.216B-parameter decoder of the checkpoint study (Section II-B,
Table I).  Only shapes are used; values come from the seeded generator.

Workloads:
  c1  one flat shard of 1,048,576 elements at offset 0; steps 1, 2, 3 chained.
  c2  one Mistral-7B MLP unit (gate, up [14336,4096], down [4096,14336]) as
      three entries of one flat allocation; steps 1 and 1000, each from the
      generated state.
  c3  146 separately allocated tensors, 152,000,000 elements, sizes drawn by
      a seeded greedy rule from {2048x2048, 512x2048, 5632x2048, 2048x5632,
      2048} with a ragged last tensor; step 10.
  c4  rank 9 of 16 of the flat Mistral-7B model (453,001,472 elements across
      2^32), one flat allocation given as 21 per-tensor pieces or 1 entry;
      step 5, then a verification digest.
  c5  the full Mistral-7B model, 291 separately allocated tensors; step 18,
      then a verification digest.
  f3  bf16-state rank shard of the 4-way sharded Mistral-7B (rank 1 of 4).
"""
from __future__ import annotations

from dataclasses import dataclass, field

from . import philox

VOCAB, D, LAYERS, KV, FFN = 32768, 4096, 32, 1024, 14336
MISTRAL_PARAMS = 7_248_023_552


@dataclass
class Piece:
    """One chunk-table entry: ``n`` elements starting at ``goff`` of the flat
    model; ``alloc`` names the allocation it lives in and ``at`` its element
    offset inside that allocation."""
    name: str
    n: int
    goff: int
    alloc: int = 0
    at: int = 0


@dataclass
class Workload:
    name: str
    pieces: list[Piece]
    steps: list[int]
    chained: bool
    verify: bool = False
    allocs: list[int] = field(default_factory=list)   # element count of each allocation

    @property
    def n(self) -> int:
        return sum(p.n for p in self.pieces)


def mistral_tensors() -> list[tuple[str, int]]:
    """(name, elements) of Mistral-7B in module registration order."""
    t = [("embed_tokens", VOCAB * D)]
    for l in range(LAYERS):
        pre = "layers.%d." % l
        t += [(pre + "q_proj", D * D), (pre + "k_proj", KV * D), (pre + "v_proj", KV * D), (pre + "o_proj", D * D),
              (pre + "gate_proj", FFN * D), (pre + "up_proj", FFN * D), (pre + "down_proj", D * FFN),
              (pre + "input_layernorm", D), (pre + "post_attention_layernorm", D)]
    t += [("norm", D), ("lm_head", VOCAB * D)]
    return t


def _separate(tensors: list[tuple[str, int]], goff0: int = 0) -> tuple[list[Piece], list[int]]:
    pieces, allocs, off = [], [], goff0
    for i, (name, n) in enumerate(tensors):
        pieces.append(Piece(name, n, off, alloc=i, at=0))
        allocs.append(n)
        off += n
    return pieces, allocs


def c1() -> Workload:
    return Workload("c1", [Piece("flat", 1 << 20, 0)], [1, 2, 3], chained=True, allocs=[1 << 20])


def c2() -> Workload:
    sizes = [("gate_proj", FFN * D), ("up_proj", FFN * D), ("down_proj", D * FFN)]
    pieces, off = [], 0
    for name, n in sizes:
        pieces.append(Piece(name, n, off, alloc=0, at=off))
        off += n
    return Workload("c2", pieces, [1, 1000], chained=False, allocs=[off])


C3_SIZES = [2048 * 2048, 512 * 2048, 5632 * 2048, 2048 * 5632, 2048]
C3_TOTAL, C3_COUNT, C3_KIND = 152_000_000, 146, 7


def c3_sizes(seed: int = 0) -> list[int]:
    """Seeded greedy draw: tensor i < 145 takes a size chosen uniformly (word
    0 of the Philox block of kind 7 at index i, modulo the count) among the
    sizes that still leave 2048 elements for every later tensor; tensor 145
    takes the remainder."""
    out, remaining = [], C3_TOTAL
    for i in range(C3_COUNT - 1):
        room = remaining - (C3_COUNT - 1 - i) * 2048
        fit = [s for s in C3_SIZES if s <= room]
        r = philox([i & 0xFFFFFFFF, i >> 32, C3_KIND << 16, 0], [seed & 0xFFFFFFFF, seed >> 32])[0]
        s = fit[r % len(fit)]
        out.append(s)
        remaining -= s
    out.append(remaining)
    assert remaining > 0 and sum(out) == C3_TOTAL
    return out


def c3(seed: int = 0) -> Workload:
    pieces, allocs = _separate([("t%d" % i, n) for i, n in enumerate(c3_sizes(seed))])
    return Workload("c3", pieces, [10], chained=False, allocs=allocs)


def rank_range(rank: int, world: int, total: int = MISTRAL_PARAMS) -> tuple[int, int]:
    return total * rank // world, total * (rank + 1) // world


def c4(rank: int = 9, world: int = 16, one_entry: bool = False) -> Workload:
    lo, hi = rank_range(rank, world)
    if one_entry:
        return Workload("c4", [Piece("shard", hi - lo, lo, 0, 0)], [5], chained=False, verify=True,
                        allocs=[hi - lo])
    pieces, off = [], 0
    for name, n in mistral_tensors():
        a, b = max(off, lo), min(off + n, hi)
        if a < b:
            pieces.append(Piece(name, b - a, a, alloc=0, at=a - lo))
        off += n
    return Workload("c4", pieces, [5], chained=False, verify=True, allocs=[hi - lo])


def c5() -> Workload:
    pieces, allocs = _separate(mistral_tensors())
    return Workload("c5", pieces, [18], chained=False, verify=True, allocs=allocs)


def f3(rank: int = 1, world: int = 4) -> Workload:
    """The paper's own per-rank shard: Mistral-7B under 4-way intra-node
    sharding (Section IV-A; 10.9 GB of BF16 state per rank, Section II-B),
    rank 1 of 4 = 1,812,005,888 elements across tensor boundaries, one flat
    allocation, bf16 state; step 5, then a verification digest."""
    w = c4(rank, world)
    w.name, w.steps = "f3", [5]
    return w


def shard(w: Workload, rank: int, world: int) -> Workload:
    """Rank ``rank``'s part of a workload under a flat-parameter (FSDP)
    partition: the contiguous range [N*r/world, N*(r+1)/world) of the
    workload's flat index range, cut from its pieces.  Each cut piece keeps
    its own allocation, of just its elements, and its global offset, so the
    digests of the ranks' shards add up to the workload's (Section II-A:
    every rank holds one contiguous range of the flattened parameters)."""
    lo0 = min(p.goff for p in w.pieces)
    lo, hi = rank_range(rank, world, w.n)
    lo, hi = lo0 + lo, lo0 + hi
    pieces, allocs = [], []
    for p in w.pieces:
        a, b = max(p.goff, lo), min(p.goff + p.n, hi)
        if a < b:
            pieces.append(Piece(p.name, b - a, a, alloc=len(allocs), at=0))
            allocs.append(b - a)
    return Workload("%s[%d/%d]" % (w.name, rank, world), pieces, list(w.steps), w.chained, w.verify, allocs)


ALL = {"c1": c1, "c2": c2, "c3": c3, "c4": c4, "c5": c5}
