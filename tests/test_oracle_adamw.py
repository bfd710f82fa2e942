"""Pins of the oracle's AdamW step and its scalar resolution.

The paper (Section III-A, Eq. 2) names the preserved state W, M, V and the
step counter but prints no update formula; the oracle takes decoupled-weight-
decay AdamW in one fixed binary32 order.  These tests pin that reading
against things other than itself:

* the scalars against exact rational arithmetic on the decimal
  hyper-parameters (within one binary32 ulp),
* the step-1 closed form (m = v = 0),
* special cases (lr = 0, g = 0, beta1 = 0, wd = 0) and non-finite inputs,
* the textbook form of AdamW evaluated in double, within a forward error
  bound derived from the number of binary32 roundings,
* the bf16 copy against torch's float -> bfloat16 conversion,
* and, informationally, torch.optim.AdamW.
"""
import math
from decimal import Decimal, getcontext
from fractions import Fraction

import numpy as np
import pytest

import oracle
import synth

EPS32 = 2.0 ** -24
HP = oracle.DEFAULT_HP
HP_DEC = dict(lr="3e-4", beta1="0.9", beta2="0.95", eps="1e-8", weight_decay="0.1")


def f32(x):
    return np.float32(x)


def ulp32(x):
    x = abs(float(x))
    return float(np.spacing(np.float32(x))) if x > 0 else 2.0 ** -149


def exact_scalars(t):
    getcontext().prec = 80
    lr, b1, b2, eps, wd = (Fraction(HP_DEC[k]) for k in ("lr", "beta1", "beta2", "eps", "weight_decay"))
    bc1 = 1 - b1 ** t
    bc2 = 1 - b2 ** t
    rs = Decimal(1) / (Decimal(bc2.numerator) / Decimal(bc2.denominator)).sqrt()
    return [b1, 1 - b1, b2, 1 - b2, eps, 1 - lr * wd, lr / bc1, Fraction(rs)]


@pytest.mark.parametrize("t", [1, 2, 3, 5, 10, 18, 1000])
def test_scalars_match_exact_rationals(t):
    got = oracle.resolve_hparams(HP, t)
    for g, e in zip(got, exact_scalars(t)):
        want = float(e)
        assert abs(float(g) - want) <= ulp32(want), (t, g, want)


def test_scalar_range_checks():
    for bad in (dict(HP, beta1=1.0), dict(HP, beta2=-0.1), dict(HP, eps=0.0), dict(HP, lr=float("nan"))):
        with pytest.raises(ValueError):
            oracle.resolve_hparams(bad, 1)
    with pytest.raises(ValueError):
        oracle.resolve_hparams(HP, 0)


def gf32(g):
    return (g.astype(np.uint32) << 16).view(np.float32)


def test_step1_closed_form():
    n = 50000
    p, _, _ = synth.state(n)
    g = synth.grad(n, step=1)
    m = np.zeros(n, np.float32)
    v = np.zeros(n, np.float32)
    h = oracle.resolve_hparams(HP, 1)
    p0 = p.copy()
    oracle.adamw(p, m, v, g, h)
    G = gf32(g)
    # m' = (1-b1) g and v' = (1-b2) g^2, each one binary32 product (g^2 of a bf16 is exact)
    assert np.array_equal(m, h[1] * G)
    assert np.array_equal(v, h[3] * (G * G))
    # p' = p (1 - lr wd) - lr g / (|g| + eps) ~ p (1 - lr wd) - lr sign(g)
    Gd = G.astype(np.float64)
    want = p0.astype(np.float64) * (1 - HP["lr"] * HP["weight_decay"]) - HP["lr"] * Gd / (np.abs(Gd) + HP["eps"])
    err = np.abs(p.astype(np.float64) - want)
    assert np.all(err <= 8 * EPS32 * (np.abs(p0) + HP["lr"]) + 1e-12)
    big = np.abs(G) > 1e-4       # |g| >> eps: the step is lr in magnitude, against the gradient's sign
    step = p0[big].astype(np.float64) * (1 - HP["lr"] * HP["weight_decay"]) - p[big]
    assert np.all(np.abs(step - HP["lr"] * np.sign(Gd[big])) < 1e-7)
    nz = G != 0                  # a zero gradient leaves only the decay
    assert np.array_equal(p[~nz], p0[~nz] * h[5])


def test_lr_zero_keeps_params():
    n = 20000
    p, m, v = synth.state(n)
    g = synth.grad(n, step=4)
    p0 = p.copy()
    h = oracle.resolve_hparams(dict(HP, lr=0.0), 4)
    assert h[5] == 1.0 and h[6] == 0.0
    oracle.adamw(p, m, v, g, h)
    assert np.array_equal(p.view(np.uint32), p0.view(np.uint32))


def test_zero_grad_decays_moments_only():
    n = 20000
    p, m, v = synth.state(n)
    m0, v0 = m.copy(), v.copy()
    g = np.zeros(n, np.uint16)
    h = oracle.resolve_hparams(HP, 7)
    oracle.adamw(p, m, v, g, h)
    assert np.array_equal(m, h[0] * m0)
    assert np.array_equal(v, h[2] * v0)


def test_beta1_zero_makes_m_the_gradient():
    n = 20000
    p, m, v = synth.state(n)
    g = synth.grad(n, step=2)
    h = oracle.resolve_hparams(dict(HP, beta1=0.0), 2)
    assert h[0] == 0.0 and h[1] == 1.0
    oracle.adamw(p, m, v, g, h)
    assert np.array_equal(m, gf32(g))


def test_weight_decay_zero():
    h = oracle.resolve_hparams(dict(HP, weight_decay=0.0), 3)
    assert h[5] == 1.0


def textbook_adamw_double(p, m, v, G, t, hp=HP):
    """Loshchilov & Hutter decoupled AdamW in double, bias corrections as
    divisions, weight decay as a separate term."""
    lr, b1, b2, eps, wd = hp["lr"], hp["beta1"], hp["beta2"], hp["eps"], hp["weight_decay"]
    p, m, v, G = (x.astype(np.float64) for x in (p, m, v, G))
    m1 = b1 * m + (1 - b1) * G
    v1 = b2 * v + (1 - b2) * G * G
    mhat = m1 / (1 - b1 ** t)
    vhat = v1 / (1 - b2 ** t)
    p1 = p - lr * (mhat / (np.sqrt(vhat) + eps) + wd * p)
    # magnitudes for the forward error bound of the binary32 evaluation
    A = np.abs(b1 * m) + np.abs((1 - b1) * G)
    den = np.sqrt(v1) / math.sqrt(1 - b2 ** t) + eps
    u = m1 / den
    step = lr / (1 - b1 ** t)
    bound_m = 3.1 * EPS32 * A
    bound_v = 3.1 * EPS32 * v1
    # subnormal m' carries an absolute rounding error (up to 2^-150 per operation) that the division by den
    # carries into u, hence the step * 2^-149 / den term
    bound_p = 1.25 * EPS32 * (2 * np.abs(p * (1 - lr * wd)) + step * (8.6 * np.abs(u) + 3.1 * A / den)
                              + np.abs(p1)) + 1.25 * step * 2.0 ** -149 / den + 2.0 ** -146
    return p1, m1, v1, bound_p, bound_m, bound_v


def adversarial_inputs(n, seed):
    rng = np.random.default_rng(seed)
    p, m, v = synth.state(n, goff=seed * n)
    g = synth.grad(n, goff=seed * n, step=seed + 1)
    k = n // 8
    # zero state, zero grad (den = eps), tiny and large gradients, denormal moments
    v[:k] = 0.0
    g[k:2 * k] = 0
    m[2 * k:3 * k] = rng.standard_normal(k).astype(np.float32) * np.float32(1e-38)
    v[2 * k:3 * k] = np.abs(rng.standard_normal(k)).astype(np.float32) * np.float32(1e-41)
    big = (rng.standard_normal(k).astype(np.float32) * np.float32(10.0)).view(np.uint32) >> 16
    g[3 * k:4 * k] = big.astype(np.uint16)
    tiny = (rng.standard_normal(k).astype(np.float32) * np.float32(1e-12)).view(np.uint32) >> 16
    g[4 * k:5 * k] = tiny.astype(np.uint16)
    p[5 * k:6 * k] = rng.standard_normal(k).astype(np.float32) * np.float32(1e-30)
    return p, m, v, g


@pytest.mark.parametrize("t", [1, 2, 3, 10, 18, 1000])
def test_against_textbook_double_within_rounding_bound(t):
    n = 80000
    p, m, v, g = adversarial_inputs(n, t)
    p1, m1, v1, bp, bm, bv = textbook_adamw_double(p, m, v, gf32(g), t)
    h = oracle.resolve_hparams(HP, t)
    oracle.adamw(p, m, v, g, h)
    assert np.all(np.abs(m - m1) <= bm + 2.0 ** -149), "m' outside the rounding bound"
    assert np.all(np.abs(v - v1) <= bv + 2.0 ** -149), "v' outside the rounding bound"
    assert np.all(np.abs(p - p1) <= bp), "p' outside the rounding bound"


def every_gradient_state(g_all):
    """Each gradient of g_all at five moment states and six parameter magnitudes."""
    states = [(0.0, 0.0), (1e-4, 1e-6), (-3e-2, 4e-5), (1e-38, 1e-41), (2.5, 7.0)]
    params = [0.0, 1e-30, -0.02, 0.7, -3.0e4, 1.0e30]
    g = np.tile(g_all, len(states) * len(params))
    m = np.repeat(np.array([s[0] for s in states], dtype=np.float32), g_all.size * len(params))
    v = np.repeat(np.array([s[1] for s in states], dtype=np.float32), g_all.size * len(params))
    p = np.tile(np.repeat(np.array(params, dtype=np.float32), g_all.size), len(states))
    return p, m, v, g


@pytest.mark.parametrize("t", [1, 18])
def test_every_bf16_gradient_within_rounding_bound(t):
    """Every bf16 gradient whose square is finite in binary32 (|g| < 2^64,
    subnormals included) against the textbook update in double, at five
    moment states and six parameter magnitudes each (1.5 million elements)."""
    g_all = np.arange(1 << 16, dtype=np.uint32).astype(np.uint16)
    g_all = g_all[(g_all & 0x7FFF) < 0x5F80]
    p, m, v, g = every_gradient_state(g_all)
    p1, m1, v1, bp, bm, bv = textbook_adamw_double(p, m, v, gf32(g), t)
    oracle.adamw(p, m, v, g, oracle.resolve_hparams(HP, t))
    assert np.all(np.abs(m - m1) <= bm + 2.0 ** -149), "m' outside the rounding bound"
    assert np.all(np.abs(v - v1) <= bv + 2.0 ** -149), "v' outside the rounding bound"
    assert np.all(np.abs(p - p1) <= bp), "p' outside the rounding bound"


def test_gradients_whose_square_overflows():
    """For finite |g| >= 2^64 the binary32 g*g overflows (IEEE: +inf), so
    v' = +inf, den = +inf, u = m'/den = 0 and p' = p*(1 - lr*wd) exactly,
    while m' stays finite and within its bound."""
    g_all = np.arange(1 << 16, dtype=np.uint32).astype(np.uint16)
    g_all = g_all[((g_all & 0x7FFF) >= 0x5F80) & ((g_all & 0x7FFF) < 0x7F80)]
    p, m, v, g = every_gradient_state(g_all)
    h = oracle.resolve_hparams(HP, 5)
    decay = np.float32(h[5])
    p_dec = p * decay
    _, m1, _, _, bm, _ = textbook_adamw_double(p, m, v, gf32(g), 5)
    oracle.adamw(p, m, v, g, h)
    assert np.all(np.isposinf(v))
    assert np.array_equal(p.view(np.uint32), p_dec.view(np.uint32))
    assert np.all(np.abs(m - m1) <= bm + 2.0 ** -149)


INF, NAN = np.float32(np.inf), np.float32(np.nan)


def test_non_finite_values_propagate_as_ieee_says():
    """One non-finite input per element, the other three finite, against what
    IEEE 754 fixes for each operation of the step (inf - inf, inf / inf and
    the square root of a negative are NaN; a finite value times a positive
    scalar keeps an infinity's sign).  The unaffected moments equal those of
    the same element with every input finite."""
    p0, m0, v0, g0 = 0.5, 0.01, 1e-4, 0x3E80          # g0 = bf16 0.25
    cases = [  # (p, m, v, g bits) -> (p', m', v') with None for "as the finite element"
        ((p0, m0, v0, 0x7F80), ("nan", INF, INF)),
        ((p0, m0, v0, 0xFF80), ("nan", -INF, INF)),
        ((p0, m0, v0, 0x7FC1), ("nan", "nan", "nan")),
        ((INF, m0, v0, g0), (INF, None, None)),
        ((-INF, m0, v0, g0), (-INF, None, None)),
        ((NAN, m0, v0, g0), ("nan", None, None)),
        ((p0, INF, v0, g0), (-INF, INF, None)),
        ((p0, -INF, v0, g0), (INF, -INF, None)),
        ((p0, NAN, v0, g0), ("nan", "nan", None)),
        ((p0, m0, INF, g0), ("decay", None, INF)),
        ((p0, m0, NAN, g0), ("nan", None, "nan")),
        ((p0, m0, -1.0, g0), ("nan", None, "negative")),
    ]
    n = len(cases) + 1
    p = np.array([c[0][0] for c in cases] + [p0], np.float32)
    m = np.array([c[0][1] for c in cases] + [m0], np.float32)
    v = np.array([c[0][2] for c in cases] + [v0], np.float32)
    g = np.array([c[0][3] for c in cases] + [g0], np.uint16)
    h = oracle.resolve_hparams(HP, 5)
    w = oracle.adamw(p, m, v, g, h)
    fin = dict(m=m[n - 1], v=v[n - 1])
    for i, (_, want) in enumerate(cases):
        for k, got, wv in (("p", p[i], want[0]), ("m", m[i], want[1]), ("v", v[i], want[2])):
            if wv is None:
                assert got.view(np.uint32) == fin[k].view(np.uint32), (i, k)
            elif wv == "nan":
                assert np.isnan(got), (i, k)
            elif wv == "decay":      # u = m' / inf = 0, so p' = p (1 - lr wd), one product
                assert got == np.float32(p0) * h[5], (i, k)
            elif wv == "negative":   # b2 v + (1 - b2) g^2 < 0: finite, and its square root is NaN
                assert np.isfinite(got) and got < 0, (i, k)
            else:
                assert got == wv, (i, k, got)
        if np.isinf(p[i]):           # the bf16 copy of an infinity is the same infinity
            assert w[i] == (0x7F80 if p[i] > 0 else 0xFF80), i


def test_bounds_would_catch_plausible_mistakes():
    """The bound is tight enough that a sign error, a dropped weight decay or
    a dropped bias correction in the oracle would fall outside it."""
    n, t = 20000, 3
    p, m, v, g = adversarial_inputs(n, 9)
    p1, _, _, bp, _, _ = textbook_adamw_double(p, m, v, gf32(g), t)
    no_wd = textbook_adamw_double(p, m, v, gf32(g), t, dict(HP, weight_decay=0.0))[0]
    assert np.mean(np.abs(no_wd - p1) > bp) > 0.8   # all but the |p| ~ 1e-30 block
    flipped = 2 * p.astype(np.float64) * (1 - HP["lr"] * HP["weight_decay"]) - p1
    assert np.mean(np.abs(flipped - p1) > bp) > 0.9
    no_bc = textbook_adamw_double(p, m, v, gf32(g), 1000)[0]
    assert np.mean(np.abs(no_bc - p1) > bp) > 0.9


def test_bf16_rounding_matches_torch():
    torch = pytest.importorskip("torch")
    hi = np.arange(1 << 16, dtype=np.uint32) << 16
    lows = np.array([0, 1, 0x3FFF, 0x7FFF, 0x8000, 0x8001, 0xC000, 0xFFFF, 0x1234, 0xABCD], dtype=np.uint32)
    u = (hi[:, None] | lows[None, :]).ravel()
    f = u.view(np.float32)
    f = f[~np.isnan(f)]
    ref = torch.from_numpy(f.copy()).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    assert np.array_equal(oracle.bf16_rne(f), ref)


def test_bf16_rounding_matches_torch_all_patterns():
    """Every one of the 2^32 binary32 bit patterns except NaNs, in chunks
    that reuse their buffers."""
    torch = pytest.importorskip("torch")
    chunk = 1 << 24
    base = np.arange(chunk, dtype=np.uint32)
    u = np.empty_like(base)
    out = torch.empty(chunk, dtype=torch.bfloat16)
    for start in range(0, 1 << 32, chunk):
        np.add(base, np.uint32(start), out=u)
        f = u.view(np.float32)
        keep = ~np.isnan(f)
        out.copy_(torch.from_numpy(f))
        ref = out.view(torch.int16).numpy().view(np.uint16)
        got = oracle.bf16_rne(f)
        assert np.array_equal(got[keep], ref[keep]), hex(start)


def test_informational_torch_adamw():
    """torch.optim.AdamW evaluates the same update in another order (lerp for
    m, division by sqrt(bc2)); both must agree within twice the rounding
    bound of the textbook form."""
    torch = pytest.importorskip("torch")
    n, t = 30000, 3
    p, m, v = synth.state(n)
    g = synth.grad(n, step=t)
    G = gf32(g)
    tp = torch.nn.Parameter(torch.from_numpy(p.copy()))
    opt = torch.optim.AdamW([tp], lr=HP["lr"], betas=(HP["beta1"], HP["beta2"]), eps=HP["eps"],
                            weight_decay=HP["weight_decay"], foreach=False)
    st = opt.state[tp]
    st["step"] = torch.tensor(float(t - 1))
    st["exp_avg"] = torch.from_numpy(m.copy())
    st["exp_avg_sq"] = torch.from_numpy(v.copy())
    tp.grad = torch.from_numpy(G.copy())
    opt.step()
    h = oracle.resolve_hparams(HP, t)
    _, _, _, bp, _, _ = textbook_adamw_double(p, m, v, G, t)
    oracle.adamw(p, m, v, g, h)
    diff = np.abs(tp.detach().numpy().astype(np.float64) - p.astype(np.float64))
    ulps = diff / np.array([ulp32(x) for x in p[:2000]] + [ulp32(x) for x in p[2000:]])
    print("torch AdamW vs oracle: max |diff| %.3g, max ulp %.1f, mean ulp %.3f" % (diff.max(), ulps.max(),
                                                                                  ulps.mean()))
    assert np.all(diff <= 2 * bp)
