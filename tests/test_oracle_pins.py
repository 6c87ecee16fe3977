"""Pins of the fp64 oracle's building blocks against what the paper and the
mathematics fix: an independent Philox implementation (numpy), a library
softmax (scipy), GetProxy's stated invariants (Algorithm 1 comments and
Sec. 5.1 constraints), Theorem 2's minimal-L1 closed form, hand-derived
examples, and the textbook special cases."""
import json
import os

import numpy as np
import pytest
from scipy.special import softmax as sp_softmax

import oracle
from oracle import enumerator as en

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _np_philox_block(counter, key):
    """Philox4x64-10 block at `counter` via numpy's implementation, which
    increments its counter before producing a block."""
    bg = np.random.Philox(key=np.asarray(key, dtype=np.uint64))
    c = [int(x) for x in counter]
    # counter - 1 with borrow across the four 64-bit words
    i = 0
    while True:
        c[i] = (c[i] - 1) % (1 << 64)
        if c[i] != (1 << 64) - 1 or i == 3:
            break
        i += 1
    st = bg.state
    st["state"]["counter"] = np.asarray(c, dtype=np.uint64)
    st["buffer_pos"] = 4
    bg.state = st
    return bg.random_raw(4)


@pytest.mark.parametrize("counter,key", [
    ([0, 0, 0, 0], [0, 0]),
    ([1, 0, 0, 0], [0, 0]),
    ([0, 0, 0, 0], [2 ** 64 - 1, 2 ** 64 - 1]),
    ([2 ** 64 - 1] * 4, [2 ** 64 - 1] * 2),
    ([7, 123456, 0, 0], [0xDEADBEEF12345678, 0]),
    ([0x243F6A8885A308D3, 0x13198A2E03707344, 0xA4093822299F31D0, 0x082EFA98EC4E6C89],
     [0x452821E638D01377, 0xBE5466CF34E90C6C]),
])
def test_philox_matches_numpy(counter, key):
    got = oracle.philox4x64_10(counter, key)
    want = _np_philox_block(counter, key)
    assert [int(x) for x in got] == [int(x) for x in want]


def test_uniform_definition():
    rng = np.random.default_rng(3)
    for _ in range(50):
        seed = int(rng.integers(0, 2 ** 63))
        seq = int(rng.integers(0, 1 << 20))
        row = int(rng.integers(0, 1 << 12))
        block = _np_philox_block([row, seq, 0, 0], [seed, 0])
        for draw in range(4):
            u = oracle.uniform(seed, seq, row, draw)
            assert u == (int(block[draw]) >> 40) / float(1 << 24)
            assert 0.0 <= u < 1.0


@pytest.mark.parametrize("T", [1.0, 0.7, 0.6, 2.5])
def test_softmax_matches_scipy(T):
    rng = np.random.default_rng(0)
    z = rng.normal(0, 4, 1000)
    z[::7] = -np.inf
    p, st = oracle.softmax(z, T)
    assert st == 0
    want = sp_softmax(np.where(np.isinf(z), -np.inf, z / T))
    np.testing.assert_allclose(p, want, rtol=1e-13, atol=1e-300)
    assert abs(p.sum() - 1) < 1e-14


def test_softmax_errors():
    z = np.array([0.0, np.nan, 1.0])
    assert oracle.softmax(z, 1.0)[1] == oracle.ERR_NONFINITE
    z = np.array([0.0, np.inf, 1.0])
    assert oracle.softmax(z, 1.0)[1] == oracle.ERR_NONFINITE
    z = np.full(5, -np.inf)
    assert oracle.softmax(z, 1.0)[1] == oracle.ERR_EMPTY_ROW


def _random_case(rng, V):
    p = sp_softmax(rng.normal(0, 2, V))
    q = sp_softmax(0.6 * np.log(p) + rng.normal(0, 1.5, V))
    return p, q


def _rejectable(rng, p, q):
    cands = np.nonzero(q > p)[0]
    return int(rng.choice(cands))


def test_get_proxy_invariants():
    """Sec. 5.1 constraints and GetProxy's comments: sum r = Z, 0 <= r <= p,
    r(x0) = 0, sum k = 1, k >= 0, k(x0) = q(x0); and the residual
    norm(max(p - k, 0)) equals r / Z."""
    rng = np.random.default_rng(1)
    for V in (2, 3, 5, 17, 64, 1000):
        for _ in range(30):
            p, q = _random_case(rng, V)
            x0 = _rejectable(rng, p, q)
            k, r, Z = oracle.get_proxy(p, q, x0)
            assert Z == pytest.approx(q[x0] - p[x0], abs=0)
            assert Z > 0
            assert abs(r.sum() - Z) < 1e-13
            assert (r >= -1e-15).all() and (r <= p + 1e-15).all()
            assert r[x0] == 0
            assert abs(k.sum() - 1) < 1e-13
            assert (k >= -1e-15).all()
            assert k[x0] == q[x0]
            R2, changed, err = oracle.reject(oracle.MODE_RESISPEC, p, q, x0)
            assert changed and err < 1e-12
            np.testing.assert_allclose(R2 * Z, r, atol=1e-15)
            # Global Mass Identity (Proposition 1): slack mass sum(k - p + r) = Z
            assert abs((k - p + r).sum() - Z) < 1e-13


@pytest.mark.parametrize("fill", [0, 1])
def test_theorem2_l1_closed_form(fill):
    """Theorem 2's proof: with capacity p (here p with p(x0) = 0, because
    GetProxy reserves nothing at x0) and budget Z, the smallest reachable
    L1(r/Z, q) is (2/Z) * sum max(0, Z q - p).  The residual of GetProxy must
    reach it, i.e. mass is added only to tokens that are not bottlenecks;
    both fills (capacity, level lam >= Z) do."""
    rng = np.random.default_rng(2)
    for V in (3, 8, 50, 500):
        for _ in range(40):
            p, q = _random_case(rng, V)
            x0 = _rejectable(rng, p, q)
            k, r, Z = oracle.get_proxy(p, q, x0, fill=fill)
            Rp = r / Z
            pt = p.copy()
            pt[x0] = 0.0
            closed = 2.0 / Z * np.maximum(0.0, Z * q - pt).sum()
            assert abs(np.abs(Rp - q).sum() - closed) < 1e-12


def test_proportional_fill_characterisation():
    """Reading R2: the deficit fills every token with capacity by the same
    fraction of that token's capacity."""
    rng = np.random.default_rng(4)
    for _ in range(40):
        p, q = _random_case(rng, 40)
        x0 = _rejectable(rng, p, q)
        k, r, Z = oracle.get_proxy(p, q, x0)
        pre = np.minimum(Z * q, p)
        pre[x0] = 0
        cap = p - pre
        cap[x0] = 0
        has = cap > 1e-9
        frac = (r[has] - pre[has]) / cap[has]
        assert frac.max() - frac.min() < 1e-10


@pytest.mark.parametrize("name", ["resispec_v3_k1.json"])
def test_golden_v3_worked_example(name):
    g = json.load(open(os.path.join(GOLDEN, name)))
    p, q = np.array(g["p"]), np.array(g["q"])
    k, r, Z = oracle.get_proxy(p, q, g["proxy_x0"])
    np.testing.assert_allclose(r, g["proxy_r"], atol=1e-15)
    np.testing.assert_allclose(k, g["proxy_K"], atol=1e-15)
    assert Z == pytest.approx(g["proxy_Z"], abs=1e-15)
    R2, _, _ = oracle.reject(oracle.MODE_RESISPEC, p, q, g["proxy_x0"])
    np.testing.assert_allclose(R2, g["residual_after_reject"], atol=1e-15)
    dist_r, _ = en.single_position(p, q, 1, en.MODE_RESISPEC)
    dist_s, _ = en.single_position(p, q, 1, en.MODE_SPECINFER)
    np.testing.assert_allclose(dist_r, g["resispec_output"], atol=1e-15)
    np.testing.assert_allclose(dist_s, g["specinfer_output"], atol=1e-15)


def test_golden_v4_clipped():
    g = json.load(open(os.path.join(GOLDEN, "resispec_proxy_v4_clipped.json")))
    p, q = np.array(g["p"]), np.array(g["q"])
    k, r, Z = oracle.get_proxy(p, q, g["x0"])
    assert Z == pytest.approx(g["Z"], abs=1e-15)
    np.testing.assert_allclose(r, g["r"], atol=1e-15)
    np.testing.assert_allclose(k, g["K"], atol=1e-15)
    R2, _, _ = oracle.reject(oracle.MODE_RESISPEC, p, q, g["x0"])
    np.testing.assert_allclose(R2, g["residual"], atol=1e-15)
    assert abs(np.abs(R2 - q).sum() - g["l1_to_q"]) < 1e-14
    # the enumerator's independent GetProxy agrees
    K2, r2, Z2 = en.proxy_resispec(p, q, g["x0"])
    np.testing.assert_allclose(r2, g["r"], atol=1e-15)


def test_golden_v4_level_fill():
    """The level reading of GetProxy's step 3 on a hand-worked case where one
    token saturates at its capacity before the level meets the budget."""
    g = json.load(open(os.path.join(GOLDEN, "resispec_proxy_v4_level_fill.json")))
    p, q = np.array(g["p"]), np.array(g["q"])
    k, r, Z = oracle.get_proxy(p, q, g["x0"], fill=oracle.FILL_LEVEL)
    assert Z == pytest.approx(g["Z"], abs=1e-15)
    np.testing.assert_allclose(r, g["r"], atol=1e-15)
    np.testing.assert_allclose(k, g["K"], atol=1e-15)
    R2, changed, err = oracle.reject(oracle.MODE_RESISPEC, p, q, g["x0"], fill=oracle.FILL_LEVEL)
    assert changed and err < 1e-14
    np.testing.assert_allclose(R2, g["residual"], atol=1e-15)
    assert abs(np.abs(R2 - q).sum() - g["l1_to_q"]) < 1e-14
    assert en.level_by_bisection(p, q, g["x0"], g["Z"]) == pytest.approx(g["level"], rel=1e-14)
    K2, r2, _ = en.proxy_resispec(p, q, g["x0"], fill=1)
    np.testing.assert_allclose(r2, g["r"], atol=1e-14)
    # the capacity fill differs on this input
    assert np.abs(oracle.get_proxy(p, q, g["x0"])[1] - r).max() > 1e-2


def test_level_fill_without_room_on_the_draft_support():
    """When r = p on the support of q cannot hold Z, the rest goes to the
    q = 0 tokens in proportion to p.  Hand-worked: p = (.1, .1, .1, .7),
    q = (.6, .4, 0, 0), x0 = 0: Z = 0.5, token 1 saturates at 0.1, the
    deficit 0.4 splits 1 : 7 over tokens 2 and 3."""
    p = np.array([0.1, 0.1, 0.1, 0.7])
    q = np.array([0.6, 0.4, 0.0, 0.0])
    k, r, Z = oracle.get_proxy(p, q, 0, fill=oracle.FILL_LEVEL)
    assert Z == pytest.approx(0.5, abs=1e-15)
    np.testing.assert_allclose(r, [0.0, 0.1, 0.05, 0.35], atol=1e-15)
    np.testing.assert_allclose(en.proxy_resispec(p, q, 0, fill=1)[1], r, atol=1e-15)


def _level_case(rng, V):
    """A rejectable case; a third of them with draft zeros."""
    p, q = _random_case(rng, V)
    if V > 3 and rng.random() < 0.33:
        z = rng.choice(V, size=max(1, V // 4), replace=False)
        q[z] = 0.0
        q /= q.sum()
    return p, q


def test_level_fill_structure():
    """fill = level: r = min(lam q, p) off x0 for one lam >= Z, sum r = Z,
    with the invariants of Sec. 5.1 (0 <= r <= p, r(x0) = 0, sum K = 1,
    K >= 0, K(x0) = q(x0)) and R' = r / Z."""
    rng = np.random.default_rng(21)
    seen = 0
    for V in (2, 3, 5, 17, 64, 1000):
        for _ in range(30):
            p, q = _level_case(rng, V)
            if not (q - p).max() > 0:
                continue
            x0 = _rejectable(rng, p, q)
            k, r, Z = oracle.get_proxy(p, q, x0, fill=oracle.FILL_LEVEL)
            assert abs(r.sum() - Z) < 1e-13
            assert (r >= -1e-15).all() and (r <= p + 1e-15).all() and r[x0] == 0
            assert abs(k.sum() - 1) < 1e-13 and (k >= -1e-15).all() and k[x0] == q[x0]
            off = np.arange(V) != x0
            if p[off & (q > 0)].sum() < Z:  # no finite level: q-support saturated
                np.testing.assert_allclose(r[off & (q > 0)], p[off & (q > 0)], atol=1e-15)
                continue
            below = off & (q > 0) & (r < p - 1e-12)
            assert (r[off & (q == 0)] == 0).all()
            if below.any():
                lam = r[below] / q[below]
                assert lam.max() - lam.min() <= 1e-11 * lam.max()
                lam = lam.mean()
                assert lam >= Z * (1 - 1e-12)
                sat = off & (q > 0) & ~below
                assert (p[sat] <= lam * q[sat] * (1 + 1e-9) + 1e-15).all()
                seen += 1
            R2, changed, err = oracle.reject(oracle.MODE_RESISPEC, p, q, x0,
                                             fill=oracle.FILL_LEVEL)
            assert changed and err < 1e-12
            np.testing.assert_allclose(R2 * Z, r, atol=1e-15)
    assert seen > 100


def test_level_fill_matches_bisection():
    """The oracle's exact level (sorted ratios) against the enumerator's
    bisection of lam -> sum min(lam q, p), an independent method."""
    rng = np.random.default_rng(22)
    for V in (3, 9, 50, 700):
        for _ in range(25):
            p, q = _level_case(rng, V)
            if not (q - p).max() > 0:
                continue
            x0 = _rejectable(rng, p, q)
            _, r, _ = oracle.get_proxy(p, q, x0, fill=oracle.FILL_LEVEL)
            _, r2, _ = en.proxy_resispec(p, q, x0, fill=1)
            np.testing.assert_allclose(r, r2, atol=1e-13)


@pytest.mark.parametrize("fill", [0, 1])
def test_binary_vocab_resispec_equals_specinfer(fill):
    """V = 2: the only token with capacity receives the whole budget, so the
    ResiSpec residual equals the SpecInfer residual (delta at the other
    token), whatever the fill."""
    rng = np.random.default_rng(5)
    for _ in range(50):
        p, q = _random_case(rng, 2)
        x0 = int(np.argmax(q - p))
        Rr, _, _ = oracle.reject(oracle.MODE_RESISPEC, p, q, x0, fill=fill)
        Rs, _, _ = oracle.reject(oracle.MODE_SPECINFER, p, q, x0)
        np.testing.assert_allclose(Rr, Rs, atol=1e-15)
        np.testing.assert_allclose(Rr, np.eye(2)[1 - x0], atol=1e-15)


def test_specinfer_reject_matches_textbook():
    rng = np.random.default_rng(6)
    for _ in range(30):
        p, q = _random_case(rng, 30)
        R2, changed, err = oracle.reject(oracle.MODE_SPECINFER, p, q, 0)
        d = np.maximum(p - q, 0)
        np.testing.assert_allclose(R2, d / d.sum(), atol=1e-15)
        assert err < 1e-14


def test_sample_matches_searchsorted():
    rng = np.random.default_rng(7)
    for V in (1, 2, 10, 1000):
        for _ in range(200):
            R = rng.random(V) * (rng.random(V) < 0.7)
            if R.sum() == 0:
                R[rng.integers(V)] = 1.0
            u = int(rng.integers(0, 1 << 24)) / float(1 << 24)
            x, m = oracle.sample(R, u)
            c = np.cumsum(R)
            want = int(np.searchsorted(c, u * c[-1], side="right"))
            assert x == want
            assert R[x] > 0
            assert 0 <= m <= 1


def test_sample_endpoints():
    R = np.array([0.0, 0.3, 0.0, 0.7, 0.0])
    assert oracle.sample(R, 0.0)[0] == 1
    assert oracle.sample(R, 1 - 2 ** -24)[0] == 3


def test_z_applied_budget_worked_examples():
    """Z_applied = max(Z*, |q(x0) - R(x0)|), Z* = min_{q>0} R/q, clamped to
    1 - R(x0) (Sec. 5.3 heuristic; the clamp keeps the water-fill feasible).
    Hand-worked cases:
      V = 2, R = (.5, .5), q = (.6, .4), reject x0 = 0: Z* = 5/6 > gap = .1,
      clamped to 1 - R(x0) = .5; r(1) = min(.5 * .4, .5) = .2, the deficit .3
      fills x1's capacity .3, so r = (0, .5) and R' = r / Z = (0, 1).
      V = 3, R = (.1, .6, .3), q = (.12, .5, .38), reject x0 = 0: Z* = .3/.38
      = 15/19 (unclamped: 1 - R(x0) = .9); r_pre = (0, 7.5/19, .3), the
      deficit 7.5/19 - .3 fills x1 (x2 has no capacity left), so r(1) =
      15/19 - .3 and R' = (0, 1 - .3 * 19/15, .3 * 19/15) = (0, .62, .38)."""
    R, q = np.array([.5, .5]), np.array([.6, .4])
    assert abs(oracle.budget(R, q, 0, 0) - 0.1) < 1e-15
    assert abs(oracle.budget(R, q, 0, 1) - 0.5) < 1e-15
    Rn, changed, err = oracle.reject(oracle.MODE_RESISPEC, R, q, 0, z_rule=1)
    assert changed and err < 1e-12
    np.testing.assert_allclose(Rn, [0.0, 1.0], atol=1e-15)
    R, q = np.array([.1, .6, .3]), np.array([.12, .5, .38])
    assert abs(oracle.budget(R, q, 0, 1) - 15 / 19) < 1e-15
    Rn, changed, err = oracle.reject(oracle.MODE_RESISPEC, R, q, 0, z_rule=1)
    assert changed and err < 1e-12
    np.testing.assert_allclose(Rn, [0.0, 0.62, 0.38], atol=1e-14)


def test_z_applied_equals_algorithm1_when_capacity_bound_is_below_gap():
    """When min_{q>0} R/q <= q(x0) - R(x0) the heuristic's max picks the gap
    and the rejection is Algorithm 1's; the bound itself is computed here
    with numpy from R and q."""
    rng = np.random.default_rng(11)
    seen = 0
    for _ in range(400):
        V = int(rng.integers(3, 40))
        R = rng.dirichlet(np.full(V, 0.7))
        q = rng.dirichlet(np.full(V, 0.7))
        x0 = int(np.argmax(q - R))
        gap = q[x0] - R[x0]
        if not (gap > 0) or np.min(R[q > 0] / q[q > 0]) > gap:
            continue
        seen += 1
        a = oracle.reject(oracle.MODE_RESISPEC, R, q, x0, z_rule=0)[0]
        b = oracle.reject(oracle.MODE_RESISPEC, R, q, x0, z_rule=1)[0]
        np.testing.assert_array_equal(a, b)
    assert seen > 100


def test_golden_fp32_error_bound_two_rejections():
    """The fp32 error bound of proxy-denominator rows (reading R11,
    oracle/fp32_error_bound.c) through two rejections, against the bound
    worked by hand in tests/golden/fp32_error_bound_v3.json (inputs there are
    exact GetProxy results, checked here against the oracle's GetProxy)."""
    g = json.load(open(os.path.join(GOLDEN, "fp32_error_bound_v3.json")))
    eps = 2.0 ** -24
    eR = oracle.fp32_error_init(g["p"])
    eD = oracle.fp32_error_init(g["q"])
    np.testing.assert_allclose(eR / eps, g["eR_init"], rtol=1e-12)
    np.testing.assert_allclose(eD / eps, g["eD_init"], rtol=1e-12)
    for j, rj in enumerate(g["rejections"], start=1):
        k, r, Z = oracle.get_proxy(rj["R"], rj["D"], rj["x0"])
        np.testing.assert_allclose(r, rj["r"], atol=1e-15)
        np.testing.assert_allclose(k, rj["K"], atol=1e-15)
        assert abs(Z - rj["Z"]) < 1e-15
        eR, eD = oracle.fp32_error_reject(rj["R"], rj["D"], rj["r"], rj["K"], rj["x0"], rj["Z"],
                                          rj["level"], rj["mu"], eR, eD)
        np.testing.assert_allclose(eR / eps, g[f"eR_after_{j}"], rtol=1e-9, atol=1e-9)
        np.testing.assert_allclose(eD / eps, g[f"eD_after_{j}"], rtol=1e-9, atol=1e-9)
