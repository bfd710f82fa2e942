"""Pins of the oracle's bf16-state step (parameters and moments stored in
bf16, the paper's setting, Section IV-A): it must equal the pinned binary32
step on the exactly widened inputs followed by torch's float -> bfloat16
rounding of p', m', v'; plus the lr = 0 special case and the digests of the
written words."""
import numpy as np
import pytest

import oracle
import synth

HP = oracle.DEFAULT_HP


def widen(h):
    return (h.astype(np.uint32) << 16).view(np.float32)


def bf16_by_torch(x):
    torch = pytest.importorskip("torch")
    return torch.from_numpy(np.ascontiguousarray(x)).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)


def edge_state(n, seed):
    rng = np.random.default_rng(seed)
    p, m, v = synth.state_bf16(n, goff=seed * n)
    g = synth.grad(n, goff=seed * n, step=seed + 1)
    k = n // 6
    v[:k] = 0
    g[:k] = 0
    m[k:2 * k] = (rng.standard_normal(k).astype(np.float32) * np.float32(1e-38)).view(np.uint32) >> 16
    g[2 * k:3 * k] = (rng.standard_normal(k).astype(np.float32) * np.float32(10.0)).view(np.uint32) >> 16
    p[3 * k:3 * k + 50] = 0x8000
    return p, m, v, g


@pytest.mark.parametrize("t", [1, 5, 1000])
def test_bf16_step_is_f32_step_then_rounding(t):
    n = 60000
    p, m, v, g = edge_state(n, t)
    h8 = oracle.resolve_hparams(HP, t)
    P, Mm, V = widen(p), widen(m), widen(v)
    oracle.adamw(P, Mm, V, g, h8)
    want = [bf16_by_torch(x) for x in (P, Mm, V)]
    oracle.adamw_bf16(p, m, v, g, h8)
    for got, exp in zip((p, m, v), want):
        assert np.array_equal(got, exp)


def test_bf16_lr_zero_keeps_params():
    p, m, v, g = edge_state(20000, 3)
    p0 = p.copy()
    oracle.adamw_bf16(p, m, v, g, oracle.resolve_hparams(dict(HP, lr=0.0), 3))
    keep = p0 != 0x8000          # -0 * 1 - 0 = +0 under round-to-nearest
    assert np.array_equal(p[keep], p0[keep])


def test_bf16_digests_are_those_of_the_written_words():
    p, m, v, g = edge_state(30001, 4)
    goff = (1 << 32) - 1000
    d = oracle.commit_bf16(p, m, v, g, goff, oracle.resolve_hparams(HP, 4))
    assert d == [oracle.digest_u16(p, goff), oracle.digest_u16(m, goff), oracle.digest_u16(v, goff)]
