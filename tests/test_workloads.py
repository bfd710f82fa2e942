"""Pins of the workload tables: the shapes, offsets and compositions that
the benchmark and the parity tests run, fixed by hand from the model
architecture and the seeded size rule, so that a change of the generator or
of the table builders cannot silently change what is measured."""
from collections import Counter

from synth import workloads as W

# Mistral-7B-v0.3: vocab 32768, d 4096, 32 layers, GQA kv 1024, FFN 14336,
# untied embedding and lm_head (arxiv 2609.18178 Section IV-A; 7,248,023,552
# parameters in the Table III caption).
PER_LAYER = 2 * 4096 * 4096 + 2 * 1024 * 4096 + 3 * 14336 * 4096 + 2 * 4096
MISTRAL_TOTAL = 2 * 32768 * 4096 + 32 * PER_LAYER + 4096


def test_mistral_parameter_count():
    assert MISTRAL_TOTAL == 7_248_023_552 == W.MISTRAL_PARAMS


def test_c5_full_model_table():
    w = W.c5()
    assert len(w.pieces) == 291 and w.n == MISTRAL_TOTAL
    names = [p.name for p in w.pieces]
    assert names[0] == "embed_tokens" and names[-2] == "norm" and names[-1] == "lm_head"
    assert names[1:10] == ["layers.0." + t for t in ("q_proj", "k_proj", "v_proj", "o_proj", "gate_proj",
                                                      "up_proj", "down_proj", "input_layernorm",
                                                      "post_attention_layernorm")]
    kinds = Counter(n.split(".")[-1] for n in names)
    assert kinds == {"embed_tokens": 1, "q_proj": 32, "k_proj": 32, "v_proj": 32, "o_proj": 32, "gate_proj": 32,
                     "up_proj": 32, "down_proj": 32, "input_layernorm": 32, "post_attention_layernorm": 32,
                     "norm": 1, "lm_head": 1}
    # one allocation per tensor, global offsets contiguous in module order
    off = 0
    for k, p in enumerate(w.pieces):
        assert p.alloc == k and p.at == 0 and p.goff == off and w.allocs[k] == p.n
        off += p.n
    assert w.steps == [18] and w.verify


def test_c4_rank_shard():
    lo, hi = W.rank_range(9, 16)
    assert (lo, hi) == (4_077_013_248, 4_530_014_720) and lo < (1 << 32) < hi
    w = W.c4()
    assert len(w.pieces) == 21 and w.n == hi - lo == 453_001_472 and w.allocs == [hi - lo]
    first, last = w.pieces[0], w.pieces[-1]
    # layer 18's k_proj starts 2,304 elements before the shard
    assert first.name == "layers.18.k_proj" and first.goff == lo and first.n == 1024 * 4096 - 2304
    assert last.name == "layers.20.o_proj" and last.n == 8_391_168 and last.goff + last.n == hi
    at = 0
    for p in w.pieces:
        assert p.at == at and p.goff == lo + at
        at += p.n
    one = W.c4(one_entry=True)
    assert len(one.pieces) == 1 and one.pieces[0].goff == lo and one.n == w.n


def test_c3_ragged_composition():
    """The seeded greedy draw over {2048x2048, 512x2048, 5632x2048,
    2048x5632, 2048}: 146 tensors whose sizes are all multiples of 2048
    except the ragged last, summing to 152,000,000."""
    sizes = W.c3_sizes()
    assert len(sizes) == 146 and sum(sizes) == 152_000_000
    assert Counter(sizes[:-1]) == {2048: 126, 11_534_336: 11, 4_194_304: 5, 1_048_576: 3}
    assert sizes[-1] == 747_008
    w = W.c3()
    assert [p.n for p in w.pieces] == sizes and w.steps == [10]


def test_c2_mlp_unit_and_c1():
    w = W.c2()
    assert [p.n for p in w.pieces] == [14336 * 4096] * 3 and [p.goff for p in w.pieces] == [0, 58_720_256,
                                                                                             117_440_512]
    assert w.n == 176_160_768 and w.allocs == [w.n] and w.steps == [1, 1000]
    c1 = W.c1()
    assert c1.n == 1 << 20 and c1.steps == [1, 2, 3] and c1.chained


def test_f3_paper_rank_shard():
    """Rank 1 of the 4-way intra-node shard of Mistral-7B (10.9 GB of BF16
    state per rank, Section II-B)."""
    w = W.f3()
    lo, hi = W.rank_range(1, 4)
    assert w.n == hi - lo == 1_812_005_888 and w.pieces[0].goff == lo and len(w.pieces) == 77
    assert w.pieces[0].name == "layers.7.up_proj" and w.pieces[-1].name == "layers.16.q_proj"
    assert 6 * w.n > 10.8e9


def test_model_split_shards_partition_the_workload():
    """Rank shards of a flat-parameter partition are contiguous, disjoint and
    cover the workload; at 16 ranks of c5, rank 9 holds c4's range in the
    same 21 pieces."""
    for w, world in ((W.c3(), 2), (W.c3(), 7), (W.c5(), 16), (W.c5(), 1)):
        lo0 = min(p.goff for p in w.pieces)
        covered = lo0
        for r in range(world):
            s = W.shard(w, r, world)
            for p in s.pieces:
                assert p.goff == covered and p.at == 0 and s.allocs[p.alloc] == p.n
                covered += p.n
            assert abs(s.n - w.n / world) <= 1
        assert covered == lo0 + w.n
    s9, c4 = W.shard(W.c5(), 9, 16), W.c4()
    assert [(p.name, p.goff, p.n) for p in s9.pieces] == [(p.name, p.goff, p.n) for p in c4.pieces]
