"""The level search the streaming kernel uses for the level fill, modelled
in numpy on the CPU: Newton steps on k from k = Z over the concave,
piecewise-linear s(k) = sum over tokens other than x0 of min(k D, R), with
the kernel's stopping rules (a deficit below 2^-22 Z, a step that no
longer moves k in fp32, 24 passes) and its normalisation by the mass
reached.  Checked against the oracle's exact level on rows with the
bench's logit distribution: the model's residual agrees with the oracle's
within the parity bound, and the passes it needs are few."""
import numpy as np
from scipy.special import softmax

import oracle

STEPS = 24


def _newton_level(R, D, x0, Z):
    """(k, passes, saturated) as the kernel takes them, sums in fp32."""
    f = np.float32
    off = np.ones(R.size, bool)
    off[x0] = False
    R32, D32, Z32 = R.astype(f), D.astype(f), f(Z)
    if R32[off & (D32 > 0)].sum(dtype=f) < Z32:   # first pass: no level reaches Z
        return np.inf, 2, True
    k = Z32
    for step in range(STEPS):
        m = np.minimum((k * D32).astype(f), R32)
        s1 = m[off].sum(dtype=f)
        slope = D32[off & (m < R32)].sum(dtype=f)
        if step + 1 >= STEPS:
            break
        gap = f(Z32 - s1)
        if not gap > Z32 * f(2.0 ** -22) or not slope > 0:
            break
        kn = f(k + gap / slope)
        if not kn > k:
            break
        k = kn
    return float(k), step + 1, False


def _bench_rows(rng, V, rho):
    ranks = rng.permutation(V) + 1
    zt = 4.0 * rng.standard_normal(V) - np.log(ranks)
    zd = rho * zt + np.sqrt(1 - rho * rho) * 4.0 * rng.standard_normal(V)
    return softmax(zt), softmax(zd)


def test_newton_level_matches_the_exact_level():
    rng = np.random.default_rng(2608)
    passes = []
    for trial in range(24):
        R, D = _bench_rows(rng, 20000, (0.5, 0.8, 0.95)[trial % 3])
        for _ in range(3):               # a chain of rejections at one node
            x0 = int(rng.choice(R.size, p=D))
            if not D[x0] > R[x0]:
                continue
            Z = D[x0] - R[x0]
            _, r, _ = oracle.get_proxy(R, D, x0, fill=oracle.FILL_LEVEL)
            exact = r / r.sum()
            k, n, sat = _newton_level(R, D, x0, Z)
            passes.append(n)
            m = np.where(np.arange(R.size) == x0, 0.0,
                         np.minimum(k * D, R) if not sat else np.where(D > 0, R, 0.0))
            model = m / m.sum()
            assert np.abs(model - exact).max() <= 1e-6
            assert np.abs(model - exact).sum() <= 1e-5
            R = exact
    passes = np.asarray(passes)
    assert passes.size >= 40
    assert passes.mean() <= 6 and passes.max() < STEPS
