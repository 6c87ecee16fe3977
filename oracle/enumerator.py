"""Exact output distribution of the verification rules, by enumeration.

TEST INFRASTRUCTURE ONLY (see ``oracle/__init__.py``).

No sampling happens here: every accept test is integrated over its uniform
analytically (accept probability min(1, R(x)/q(x)), Sec. 3), and every
candidate value is summed over with its draft probability q(x) (candidates
are i.i.d. draws from q, Sec. 4).  The cost is V**k per node with k
candidates, so this is for tiny vocabularies only.

The shaping rules are written here a second time, independently of the C
oracle and vectorised over the vocabulary:

* SPECINFER: R' = (R - q)_+ / sum (R - q)_+                    (Eq. 2, Sec. 3)
* RESISPEC:  GetProxy of Algorithm 1 with budget Z = q(x0) - R(x0),
  projection r = min(Z q, R) with r(x0) = 0, the deficit filled in
  proportion to the remaining capacity R - r off x0, then
  R' = norm(max(R - K, 0)) with K = R - r and K(x0) = q(x0).
* RESISPEC with the proxy as the next test denominator (the paper's EAGLE
  integration, App. C): after each rejection the denominator D used by the
  accept tests and by the next GetProxy becomes that rejection's K; the
  candidates are still drawn from the draft q.
* RESISPEC with the Z_applied budget (``z_rule=1``, the Sec. 5.3 heuristic):
  Z = max(Z*, |q(x0) - R(x0)|) with Z* the smallest R/q over q > 0, at most
  1 - R(x0).
* RESISPEC with the level fill (``fill=1``): r = min(lam q, R) off x0 with
  the level lam >= Z that makes sum r = Z, found here by bisection on the
  nondecreasing function lam -> sum min(lam q, R) (the C oracle solves it
  exactly on the sorted ratios instead); when no finite level reaches Z,
  r = R on the support of q and the tokens with q = 0 take the rest in
  proportion to R.
"""
from __future__ import annotations

from functools import lru_cache

import numpy as np

MODE_RESISPEC = 0
MODE_SPECINFER = 1


def shape_specinfer(R, q, x0=None):
    d = np.maximum(R - q, 0.0)
    s = d.sum()
    return R.copy() if not s > 0 else d / s


def level_by_bisection(R, q, x0, Z, iters=200):
    """The level lam with sum_{x != x0} min(lam q, R) = Z, or inf when the
    support of q cannot hold Z."""
    w = np.ones(R.size, dtype=bool)
    w[x0] = False
    f = lambda lam: float(np.minimum(lam * q[w], R[w]).sum())
    if R[w & (q > 0)].sum() < Z:
        return np.inf
    lo, hi = 0.0, 1.0
    while f(hi) < Z:
        hi *= 2.0
    for _ in range(iters):
        mid = 0.5 * (lo + hi)
        if f(mid) < Z:
            lo = mid
        else:
            hi = mid
        if hi - lo <= 4e-16 * hi:
            break
    return hi


def budget(R, q, x0, z_rule=0):
    gap = q[x0] - R[x0]
    if z_rule == 0:
        return gap
    zstar = np.min(R[q > 0] / q[q > 0])
    return min(max(zstar, abs(gap)), 1.0 - R[x0])


def proxy_resispec(R, q, x0, fill=0, z_rule=0):
    """Returns (K, r, Z) of GetProxy(R, q, x0)."""
    Z = budget(R, q, x0, z_rule)
    lam = Z if fill == 0 else level_by_bisection(R, q, x0, Z)
    r = np.minimum(lam * q, R) if np.isfinite(lam) else np.where(q > 0, R, 0.0)
    r[x0] = 0.0
    cap = R - r
    cap[x0] = 0.0
    deficit = Z - r.sum()
    if cap.sum() > 0 and (fill == 0 or not np.isfinite(lam)):
        r = r + deficit * cap / cap.sum()
    K = R - r
    K[x0] = q[x0]
    return K, r, Z


def shape_resispec(R, q, x0, fill=0, z_rule=0):
    K, r, Z = proxy_resispec(R, q, x0, fill, z_rule)
    if not Z > 0:
        return R.copy()
    d = np.maximum(R - K, 0.0)
    s = d.sum()
    return R.copy() if not s > 0 else d / s


def shape(mode, R, q, x0, fill=0, z_rule=0):
    return (shape_specinfer(R, q) if mode == MODE_SPECINFER
            else shape_resispec(R, q, x0, fill, z_rule))


def accept_prob(R, D, x):
    """P(u D(x) < R(x)) for u ~ U[0, 1)."""
    if D[x] > 0:
        return min(1.0, R[x] / D[x])
    return 1.0 if R[x] > 0 else 0.0


def reject_step(mode, R, D, x, denom_update, fill=0, z_rule=0):
    """(R', D') after candidate x is rejected."""
    if mode == MODE_SPECINFER or not denom_update:
        return shape(mode, R, D, x, fill, z_rule), D
    K, r, Z = proxy_resispec(R, D, x, fill, z_rule)
    if not Z > 0:
        return R.copy(), D
    d = np.maximum(R - K, 0.0)
    s = d.sum()
    if not s > 0:
        return R.copy(), D
    return d / s, K


def single_position(p, q, k, mode, denom_update=False, fill=0, z_rule=0):
    """Exact distribution of the emitted token when k i.i.d. candidates from q
    are tested in order against the residual chain starting at p, with the
    residual sample after k rejections (``denom_update``: the test
    denominator becomes each rejection's proxy, ResiSpec mode).

    Returns (dist, accept_prob_by_position) where accept_prob_by_position[i]
    is P(candidate i+1 is the accepted one).
    """
    p = np.asarray(p, dtype=np.float64)
    q = np.asarray(q, dtype=np.float64)
    V = p.size
    acc = np.zeros(k)

    def rec(R, D, m, weight, depth):
        out = np.zeros(V)
        if m == 0:
            return R.copy()
        for x in range(V):
            if q[x] <= 0:
                continue
            a = accept_prob(R, D, x)
            out[x] += q[x] * a
            acc[depth] += weight * q[x] * a
            if a < 1.0:
                R2, D2 = reject_step(mode, R, D, x, denom_update, fill, z_rule)
                out += q[x] * (1.0 - a) * rec(R2, D2, m - 1, weight * q[x] * (1.0 - a),
                                              depth + 1)
        return out

    dist = rec(p.copy(), q.copy(), k, 1.0, 0)
    return dist, acc


def tree_walk(parents, rows, mode, fill=0):
    """Exact distribution over emitted token tuples for a draft tree.

    ``parents``: int [N] (parent < child, -1 = root).  ``rows(path)`` returns
    (p, q) for the node reached by the token tuple ``path`` (rows depend on
    the path only, so duplicate siblings share rows as a real model would).
    The emitted tuple is the accepted tokens followed by the residual (all
    children rejected) or bonus (accepted node without children) token.
    Returns {tuple: probability}.
    """
    parents = list(int(x) for x in parents)
    kids = {n: [c for c, pa in enumerate(parents) if pa == n]
            for n in [-1] + list(range(len(parents)))}

    @lru_cache(maxsize=None)
    def visit(node, path):
        p, q = rows(path)
        p = np.asarray(p, dtype=np.float64)
        q = np.asarray(q, dtype=np.float64)
        ch = kids[node]
        if not ch:
            return {(y,): float(p[y]) for y in range(p.size) if p[y] > 0}

        def rec(R, j):
            out = {}
            if j == len(ch):
                for y in range(R.size):
                    if R[y] > 0:
                        out[(y,)] = out.get((y,), 0.0) + float(R[y])
                return out
            c = ch[j]
            for x in range(q.size):
                if q[x] <= 0:
                    continue
                a = min(1.0, R[x] / q[x])
                if a > 0:
                    for seq, pr in visit(c, path + (x,)).items():
                        key = (x,) + seq
                        out[key] = out.get(key, 0.0) + q[x] * a * pr
                if a < 1.0:
                    R2 = shape(mode, R, q, x, fill)
                    for seq, pr in rec(R2, j + 1).items():
                        out[seq] = out.get(seq, 0.0) + q[x] * (1.0 - a) * pr
            return out

        return rec(p.copy(), 0)

    return visit(-1, ())
