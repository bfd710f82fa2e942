"""Pins of the oracle's state digest.

D_B = sum_i splitmix64(((G_i mod 2^32) << 32) | bits_B(i)) mod 2^64, with
splitmix64(x) the first SplitMix64 output for seed x.  The pins are the
published SplitMix64 seed-0 stream, and properties of the definition:
concatenation, chunking invariance, bijectivity of the mix (so any one changed
element changes the digest), index-swap detection, zero-extension of bf16 words,
and the 2^32 period of the index key.
"""
import numpy as np
import pytest

import oracle
from conftest import read_golden

GAMMA = 0x9E3779B97F4A7C15
M64 = (1 << 64) - 1


def kat():
    return [int(r[0], 16) for r in read_golden("splitmix64_seed0_stream.txt")]


def test_splitmix64_published_stream():
    # output k of the seed-0 SplitMix64 stream is splitmix64(k * gamma)
    for k, want in enumerate(kat()):
        assert oracle.splitmix64((k * GAMMA) & M64) == want


def test_single_element_digest_uses_index_high_bits_high():
    """A one-element digest at global index G with word b is splitmix64 of the
    key (G << 32) | b: taking keys from the published stream pins the key
    layout (index in the high half, bits in the low half)."""
    for k, want in enumerate(kat()):
        key = (k * GAMMA) & M64
        G, b = key >> 32, key & 0xFFFFFFFF
        assert oracle.digest_f32(np.array([b], dtype=np.uint32), goff=G) == want
    # G = 0 and a zero word: the seed-0 first output, through both word widths
    assert oracle.digest_u16(np.zeros(1, np.uint16), 0) == kat()[0]
    assert oracle.digest_f32(np.zeros(1, np.uint32), 0) == kat()[0]


def test_digest_is_wrapping_sum_of_element_digests():
    """Brute force on <= 64 elements: the digest of a buffer equals the
    wrapping sum of its one-element digests at the right global indices."""
    rng = np.random.default_rng(1)
    special = np.array([0, 1, 0x80000000, 0x7F800000, 0xFF800000, 0x00000001, 0x807FFFFF, 0xFFFFFFFF],
                       dtype=np.uint32)
    for goff in (0, 17, (1 << 32) - 5, (1 << 32) + 3, (1 << 40) - 1, M64 - 40):
        for n in (1, 2, 7, 8, 9, 31, 64):
            bits = rng.integers(0, 2**32, size=n, dtype=np.uint64).astype(np.uint32)
            bits[: min(n, len(special))] = special[: min(n, len(special))]
            want = 0
            for i in range(n):
                want = (want + oracle.digest_f32(bits[i:i + 1], (goff + i) & M64)) & M64
            assert oracle.digest_f32(bits, goff) == want


def test_concatenation_and_chunking():
    rng = np.random.default_rng(2)
    a = rng.integers(0, 2**32, size=1000, dtype=np.uint64).astype(np.uint32)
    o = (1 << 32) - 600            # straddles 2^32
    whole = oracle.digest_f32(a, o)
    for cut in (0, 1, 599, 600, 601, 999, 1000):
        assert (oracle.digest_f32(a[:cut], o) + oracle.digest_f32(a[cut:], o + cut)) & M64 == whole
    cuts = sorted(rng.choice(np.arange(1, 1000), size=20, replace=False).tolist())
    parts, prev = 0, 0
    for c in cuts + [1000]:
        parts = (parts + oracle.digest_f32(a[prev:c], o + prev)) & M64
        prev = c
    assert parts == whole


def test_bf16_words_are_zero_extended():
    rng = np.random.default_rng(3)
    h = rng.integers(0, 2**16, size=257, dtype=np.uint64).astype(np.uint16)
    assert oracle.digest_u16(h, 12345) == oracle.digest_f32(h.astype(np.uint32), 12345)


def test_any_single_bit_flip_changes_digest():
    """splitmix64 is a bijection of 64-bit words (odd multiplies and
    xor-right-shifts are invertible), so changing one element's word always
    changes its term and hence the sum."""
    rng = np.random.default_rng(4)
    a = rng.integers(0, 2**32, size=512, dtype=np.uint64).astype(np.uint32)
    base = oracle.digest_f32(a, 77)
    for pos in (0, 1, 255, 511):
        for bit in range(32):
            b = a.copy()
            b[pos] ^= np.uint32(1 << bit)
            assert oracle.digest_f32(b, 77) != base
    h = a.astype(np.uint16)
    base16 = oracle.digest_u16(h, 77)
    for bit in range(16):
        g = h.copy()
        g[3] ^= np.uint16(1 << bit)
        assert oracle.digest_u16(g, 77) != base16


def test_index_swap_of_unequal_values_changes_digest():
    rng = np.random.default_rng(5)
    a = rng.integers(0, 2**32, size=300, dtype=np.uint64).astype(np.uint32)
    base = oracle.digest_f32(a, (1 << 32) - 100)
    for _ in range(200):
        i, j = rng.choice(300, size=2, replace=False)
        if a[i] == a[j]:
            continue
        b = a.copy()
        b[i], b[j] = a[j], a[i]
        assert oracle.digest_f32(b, (1 << 32) - 100) != base


def test_index_key_has_period_2_32():
    """Only G mod 2^32 enters the key: the same words 2^32 positions apart
    digest identically (a documented property of the definition)."""
    rng = np.random.default_rng(6)
    a = rng.integers(0, 2**32, size=100, dtype=np.uint64).astype(np.uint32)
    assert oracle.digest_f32(a, 5) == oracle.digest_f32(a, 5 + (1 << 32)) == oracle.digest_f32(a, 5 + (7 << 32))
    assert oracle.digest_f32(a, 5) != oracle.digest_f32(a, 6)


def test_zero_buffer():
    z = np.zeros(50, dtype=np.uint32)
    want = 0
    for i in range(50):
        want = (want + oracle.splitmix64(((1000 + i) & 0xFFFFFFFF) << 32)) & M64
    assert oracle.digest_f32(z, 1000) == want


def test_threaded_commit_matches_single_thread():
    import synth
    n = 100003
    h8 = oracle.resolve_hparams(oracle.DEFAULT_HP, 3)
    outs = []
    for nt in (1, 5):
        p, m, v = synth.state(n, goff=(1 << 32) - 50000)
        g = synth.grad(n, goff=(1 << 32) - 50000, step=3)
        w, d = oracle.commit(p, m, v, g, (1 << 32) - 50000, h8, nthreads=nt)
        outs.append((p, m, v, w, d))
    a, b = outs
    for x, y in zip(a[:4], b[:4]):
        assert np.array_equal(x.view(np.uint8), y.view(np.uint8))
    assert a[4] == b[4]
    # and the fused digests are the digests of the written buffers
    p, m, v, w, d = a
    goff = (1 << 32) - 50000
    assert d == [oracle.digest_f32(p, goff), oracle.digest_f32(m, goff), oracle.digest_f32(v, goff),
                 oracle.digest_u16(w, goff)]
