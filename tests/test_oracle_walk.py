"""The oracle's full verification walk pinned against the exact enumerator,
the textbook exactness of multi-candidate speculative sampling (Sec. 3,
Eq. 2), closed forms, independent recomputations with numpy/scipy and
the error contract."""
import numpy as np
import pytest
from scipy.special import softmax as sp_softmax
from scipy.stats import chi2

import oracle
from oracle import enumerator as en
from paper_2608_24411_gb300 import workloads as W


def chisq_pvalue(counts, probs, min_expected=5.0):
    """Pearson chi-square with bins merged (in descending expected order)
    until each expected count is >= min_expected."""
    counts = np.asarray(counts, dtype=np.float64)
    n = counts.sum()
    exp = np.asarray(probs, dtype=np.float64) * n
    assert np.all(counts[exp == 0] == 0), "mass observed where none is expected"
    order = np.argsort(-exp)
    c_bins, e_bins = [], []
    acc_c = acc_e = 0.0
    for i in order:
        acc_c += counts[i]
        acc_e += exp[i]
        if acc_e >= min_expected:
            c_bins.append(acc_c)
            e_bins.append(acc_e)
            acc_c = acc_e = 0.0
    if acc_e > 0 and e_bins:
        c_bins[-1] += acc_c
        e_bins[-1] += acc_e
    c_bins, e_bins = np.array(c_bins), np.array(e_bins)
    stat = ((c_bins - e_bins) ** 2 / e_bins).sum()
    dof = max(1, len(e_bins) - 1)
    return float(chi2.sf(stat, dof)), len(e_bins)


def _pq(seed, V, scale=1.5, rho=0.5):
    rng = np.random.default_rng(seed)
    zt = scale * rng.standard_normal(V)
    zd = rho * zt + np.sqrt(1 - rho * rho) * scale * rng.standard_normal(V)
    return zt.astype(np.float32), zd.astype(np.float32)


# ------------------------------------------------------------ enumerator pins


@pytest.mark.parametrize("V,k", [(2, 1), (3, 2), (4, 3), (6, 2), (5, 4)])
def test_enumerator_specinfer_is_exact(V, k):
    """Multi-candidate sequential verification with the residual recurrence
    reproduces p exactly (the textbook property the paper relies on)."""
    for s in range(5):
        zt, zd = _pq(100 * V + s, V)
        p, q = sp_softmax(zt.astype(np.float64)), sp_softmax(zd.astype(np.float64))
        dist, acc = en.single_position(p, q, k, en.MODE_SPECINFER)
        np.testing.assert_allclose(dist, p, atol=1e-13)
        # k = 1 closed form: P(accept) = sum min(p, q)
        _, acc1 = en.single_position(p, q, 1, en.MODE_SPECINFER)
        assert abs(acc1[0] - np.minimum(p, q).sum()) < 1e-14


def test_enumerator_resispec_special_cases():
    rng = np.random.default_rng(9)
    for _ in range(10):
        p = sp_softmax(rng.normal(0, 1, 2))
        q = sp_softmax(rng.normal(0, 1, 2))
        for k in (1, 2, 3):
            dist, _ = en.single_position(p, q, k, en.MODE_RESISPEC)
            np.testing.assert_allclose(dist, p, atol=1e-14)  # V = 2 reduces to SpecInfer
    p = sp_softmax(rng.normal(0, 1, 5))
    dist, acc = en.single_position(p, p, 3, en.MODE_RESISPEC)
    np.testing.assert_allclose(dist, p, atol=1e-15)           # q = p never rejects
    assert acc[0] == pytest.approx(1.0, abs=1e-15)


def test_resispec_output_is_biased():
    """Finding: Algorithm 1 as written is not distribution-exact (the proxy
    depends on the rejected candidate, which Theorem 1's argument does not
    allow).  The enumerated output differs from p by a clear margin."""
    tvs = []
    for s in range(6):
        zt, zd = _pq(700 + s, 6, scale=2.0, rho=0.5)
        p, q = sp_softmax(zt.astype(np.float64)), sp_softmax(zd.astype(np.float64))
        dist, _ = en.single_position(p, q, 3, en.MODE_RESISPEC)
        assert abs(dist.sum() - 1) < 1e-13
        tvs.append(0.5 * np.abs(dist - p).sum())
    assert min(tvs) > 1e-3, tvs


def test_tree_enumerator_joint_exactness_specinfer():
    """Two levels, rows a function of the token path: the first emitted token
    follows p_root and the second, given the first was an accepted candidate,
    follows p(. | first)."""
    parents = W.tree_levels([2, 2])
    V = 4
    rows_z = W.path_rows_np(11, V, 1.0, 0.5)
    T = 1.0

    def rows(path):
        zt, zd = rows_z(path)
        return sp_softmax(zt.astype(np.float64) / T), sp_softmax(zd.astype(np.float64) / T)

    dist = en.tree_walk(parents, rows, en.MODE_SPECINFER)
    assert abs(sum(dist.values()) - 1) < 1e-13
    p_root = rows(())[0]
    first = np.zeros(V)
    for seq, pr in dist.items():
        first[seq[0]] += pr
    np.testing.assert_allclose(first, p_root, atol=1e-13)
    for y1 in range(V):
        cond = np.zeros(V)
        for seq, pr in dist.items():
            if len(seq) >= 2 and seq[0] == y1:
                cond[seq[1]] += pr
        if cond.sum() > 0:
            np.testing.assert_allclose(cond / cond.sum(), rows((y1,))[0], atol=1e-12)


# ------------------------------------------------------------ oracle vs enumerator


def _single_position_draws(seed, V, k, n, zt, zd, T=1.0):
    """n independent draws (fresh candidates each) of one single-position
    problem, with the rows shared across draws (seq_stride = 0)."""
    rng = np.random.default_rng(seed)
    q = sp_softmax(zd.astype(np.float64) / T)
    cand = rng.choice(V, size=(n, k), p=q).astype(np.int32)
    target = np.ascontiguousarray(np.broadcast_to(zt, (k + 1, V)), dtype=np.float32)
    draft = np.ascontiguousarray(np.broadcast_to(zd, (k + 1, V)), dtype=np.float32)
    return target, draft, cand


@pytest.mark.parametrize("mode,fill", [(oracle.MODE_SPECINFER, 0), (oracle.MODE_RESISPEC, 0),
                                       (oracle.MODE_RESISPEC, oracle.FILL_LEVEL)])
def test_oracle_matches_enumerator_single_position(mode, fill):
    V, k, n = 8, 3, 400_000
    zt, zd = _pq(42, V, scale=1.5, rho=0.4)
    target, draft, cand = _single_position_draws(5, V, k, n, zt, zd)
    out = oracle.verify(target, draft, W.tree_single(k), cand, 1.0, seed=1234, mode=mode,
                        seq_stride=0, check_invariants=True, fill=fill)
    assert (out["status"] & ~oracle.INFO_DEGENERATE == 0).all()
    assert out["inv_err"].max() < 1e-12
    y = out["tokens"][:, 0]          # first emitted token (accepted or residual)
    p = sp_softmax(zt.astype(np.float64))
    q = sp_softmax(zd.astype(np.float64))
    dist, acc = en.single_position(p, q, k, mode, fill=fill)
    pv, nb = chisq_pvalue(np.bincount(y, minlength=V), dist)
    assert pv > 1e-4, (pv, nb)
    if fill:  # a different law from the capacity fill's (close to it on this input)
        assert 0.5 * np.abs(dist - en.single_position(p, q, k, mode)[0]).sum() > 1e-5
    # which candidate got accepted: enumerated per-position probabilities
    which = np.bincount(out["accept_len"] * 0 + np.where(out["accept_len"] > 0,
                                                         out["nodes"][:, 0], k), minlength=k + 1)
    probs = np.append(acc, 1 - acc.sum())
    pv2, _ = chisq_pvalue(which, probs)
    assert pv2 > 1e-4
    if mode == oracle.MODE_SPECINFER:
        np.testing.assert_allclose(dist, p, atol=1e-13)


def test_oracle_specinfer_million_draws_vs_target():
    """>= 1e6 draws: the SpecInfer-mode oracle output does not reject p."""
    V, k, n = 64, 3, 1_000_000
    zt, zd = _pq(77, V, scale=2.0, rho=0.8)
    target, draft, cand = _single_position_draws(8, V, k, n, zt, zd)
    out = oracle.verify(target, draft, W.tree_single(k), cand, 1.0, seed=99,
                        mode=oracle.MODE_SPECINFER, seq_stride=0)
    y = out["tokens"][:, 0]          # first emitted token (accepted or residual)
    p = sp_softmax(zt.astype(np.float64))
    pv, nb = chisq_pvalue(np.bincount(y, minlength=V), p)
    assert pv > 1e-4, (pv, nb)


def test_oracle_resispec_million_draws_rejects_target():
    """The same 1e6-draw test on the ResiSpec-mode oracle rejects p (the
    documented bias) and does not reject the enumerated output law."""
    V, k, n = 16, 3, 1_000_000
    zt, zd = _pq(78, V, scale=2.0, rho=0.8)
    target, draft, cand = _single_position_draws(9, V, k, n, zt, zd)
    out = oracle.verify(target, draft, W.tree_single(k), cand, 1.0, seed=7,
                        mode=oracle.MODE_RESISPEC, seq_stride=0)
    y = out["tokens"][:, 0]          # first emitted token (accepted or residual)
    counts = np.bincount(y, minlength=V)
    p = sp_softmax(zt.astype(np.float64))
    q = sp_softmax(zd.astype(np.float64))
    dist, _ = en.single_position(p, q, k, en.MODE_RESISPEC)
    pv_alg, _ = chisq_pvalue(counts, dist)
    pv_p, _ = chisq_pvalue(counts, p)
    assert pv_alg > 1e-4
    assert pv_p < 1e-12
    assert 0.5 * np.abs(dist - p).sum() > 1e-2


@pytest.mark.parametrize("mode,fill", [(oracle.MODE_SPECINFER, 0), (oracle.MODE_RESISPEC, 0),
                                       (oracle.MODE_RESISPEC, oracle.FILL_LEVEL)])
def test_oracle_tree_walk_matches_enumerator(mode, fill):
    """Two-level tree with path-consistent rows: the oracle's emitted
    (first, second) token pairs follow the enumerated joint law."""
    parents = W.tree_levels([2, 2])
    V, B, T = 4, 60_000, 1.0
    target, draft, cand, rows_z = W.make_path_inputs_np(21, parents, B, V, T,
                                                        scale=1.0, rho=0.5)
    out = oracle.verify(target, draft, parents, cand, T, seed=5, mode=mode, fill=fill)
    assert (out["status"] & ~oracle.INFO_DEGENERATE == 0).all()

    def rows(path):
        zt, zd = rows_z(path)
        return sp_softmax(zt.astype(np.float64) / T), sp_softmax(zd.astype(np.float64) / T)

    dist = en.tree_walk(parents, rows, mode, fill=fill)
    keys = sorted(dist)
    index = {kk: i for i, kk in enumerate(keys)}
    counts = np.zeros(len(keys))
    for b in range(B):
        a = out["accept_len"][b]
        seq = tuple(int(t) for t in out["tokens"][b, :a + 1])
        counts[index[seq]] += 1
    pv, nb = chisq_pvalue(counts, np.array([dist[kk] for kk in keys]))
    assert pv > 1e-4, (pv, nb)


# ------------------------------------------------------------ independent recomputation


def _searchsorted_draw(R, u):
    c = np.cumsum(R)
    return int(np.searchsorted(c, u * c[-1], side="right"))


def _np_uniform(seed, seq, row, draw):
    from tests.test_oracle_pins import _np_philox_block
    return (int(_np_philox_block([row, seq, 0, 0], [seed, 0])[draw]) >> 40) / float(1 << 24)


def test_identical_rows_accept_everything():
    """q = p: every first candidate is accepted, the walk follows the first
    child at every level, and the bonus is drawn from the leaf's p."""
    parents = W.tree_levels([3, 2, 2])
    V, B, T = 50, 40, 0.8
    rng = np.random.default_rng(3)
    z = rng.normal(0, 2, (B, parents.size + 1, V)).astype(np.float32)
    cand = rng.integers(0, V, (B, parents.size)).astype(np.int32)
    out = oracle.verify(z, z.copy(), parents, cand, T, seed=17, mode=oracle.MODE_RESISPEC)
    path = [0, 3, 9]           # first child at each level (BFS numbering)
    for b in range(B):
        assert out["accept_len"][b] == 3
        assert list(out["nodes"][b]) == path
        assert list(out["tokens"][b, :3]) == [cand[b, c] for c in path]
        p_leaf = sp_softmax(z[b, path[-1] + 1].astype(np.float64) / np.float32(T))
        u = _np_uniform(17, b, path[-1] + 1, 1)
        assert out["tokens"][b, 3] == _searchsorted_draw(p_leaf, u)
        assert out["rejects"][b] == 0
        assert out["rows"][b] == 2 * 3 + 1


@pytest.mark.parametrize("mode", [oracle.MODE_SPECINFER, oracle.MODE_RESISPEC])
def test_impossible_candidates_reject_everything(mode):
    """Candidates on tokens the target masks (-inf) are always rejected; the
    residual after all rejections matches the enumerator's own shaping chain
    and the final draw matches numpy's searchsorted."""
    parents = W.tree_single(4)
    V, B = 30, 25
    rng = np.random.default_rng(8)
    zt = rng.normal(0, 2, (B, 5, V)).astype(np.float32)
    zd = rng.normal(0, 2, (B, 5, V)).astype(np.float32)
    cand = rng.integers(0, 10, (B, 4)).astype(np.int32)
    zt[:, :, :10] = -np.inf
    out = oracle.verify(zt, zd, parents, cand, 1.0, seed=3, mode=mode, want_dist=True,
                        check_invariants=True)
    assert (out["accept_len"] == 0).all()
    assert out["inv_err"].max() < 1e-12
    for b in range(B):
        R = sp_softmax(np.where(np.isinf(zt[b, 0]), -np.inf, zt[b, 0].astype(np.float64)))
        q = sp_softmax(zd[b, 0].astype(np.float64))
        for x in cand[b]:
            R = en.shape(mode, R, q, int(x))
        np.testing.assert_allclose(out["dist"][b], R, atol=1e-13)
        u = _np_uniform(3, b, 0, 1)
        assert out["tokens"][b, 0] == _searchsorted_draw(R, u)


def test_shared_rows_equal_explicit_rows():
    w = W.WORKLOADS["tiny-chain-v64"]
    inp = W.make_inputs_np(w, seed=1, batch=1)
    B = 50
    rng = np.random.default_rng(2)
    cand = rng.integers(0, 64, (B, w.num_nodes)).astype(np.int32)
    shared = oracle.verify(inp["target"][0], inp["draft"][0], inp["parents"], cand, 1.0, 5,
                           seq_stride=0)
    full = oracle.verify(np.repeat(inp["target"], B, 0), np.repeat(inp["draft"], B, 0),
                         inp["parents"], cand, 1.0, 5)
    for k in ("tokens", "accept_len", "nodes", "rejects"):
        np.testing.assert_array_equal(shared[k], full[k])


def test_bf16_bits_equal_float_values():
    w = W.WORKLOADS["tree60-v32000"]
    inp = W.make_inputs_np(w, seed=3, batch=1)
    a = oracle.verify(inp["target"], inp["draft"], inp["parents"], inp["cand"], 1.0, 9,
                      want_dist=True)
    b = oracle.verify(W.bf16_bits_to_f32(inp["target"]), W.bf16_bits_to_f32(inp["draft"]),
                      inp["parents"], inp["cand"], 1.0, 9, want_dist=True)
    for k in ("tokens", "accept_len", "nodes", "dist"):
        np.testing.assert_array_equal(a[k], b[k])


def test_error_contract():
    parents = W.tree_levels([2, 2])
    V, B = 16, 6
    rng = np.random.default_rng(1)
    zt = rng.normal(0, 1, (B, 7, V)).astype(np.float32)
    zd = zt.copy()
    cand = rng.integers(0, V, (B, 6)).astype(np.int32)
    cand[1, 0] = V                     # token out of range
    zt[2, 0, 3] = np.nan               # non-finite logit in a visited row
    zt[3, 0, :] = -np.inf              # all -inf row
    zt[4, 6, 0] = np.nan               # row of a node that is never visited
    out = oracle.verify(zt, zd, parents, cand, 1.0, 0, max_depth=2)
    assert out["status"][0] == 0 and out["accept_len"][0] == 2
    assert out["status"][1] == oracle.ERR_TOKEN and out["accept_len"][1] == -1
    assert out["status"][2] == oracle.ERR_NONFINITE and out["accept_len"][2] == -1
    assert out["status"][3] == oracle.ERR_EMPTY_ROW
    assert out["status"][4] == 0
    assert (out["tokens"][1:4] == -1).all()
    depth_err = oracle.verify(zt[:1], zd[:1], parents, cand[:1], 1.0, 0, max_depth=1)
    assert depth_err["status"][0] == oracle.ERR_DEPTH
    bad_tree = np.array([-1, 1, 0, 0, 1, 1], dtype=np.int32)   # node 1 is its own parent
    bt = oracle.verify(zt[:1], zd[:1], bad_tree, cand[:1], 1.0, 0, max_depth=3)
    assert bt["status"][0] == oracle.ERR_TREE


def test_empty_tree_samples_root():
    V, B = 12, 30
    rng = np.random.default_rng(4)
    zt = rng.normal(0, 1, (B, 1, V)).astype(np.float32)
    out = oracle.verify(zt, zt, np.zeros(0, np.int32), np.zeros((B, 0), np.int32), 1.0, 6)
    assert (out["accept_len"] == 0).all()
    for b in range(B):
        p = sp_softmax(zt[b, 0].astype(np.float64))
        assert out["tokens"][b, 0] == _searchsorted_draw(p, _np_uniform(6, b, 0, 1))


def test_per_sequence_trees_equal_separate_shared_tree_calls():
    """A [B, N] parents call (a tree per sequence) equals B calls that each
    pass that sequence's tree as the shared tree (the path the other pins
    cover), with the sequence's index for the draws; a bad tree marks only
    its own sequence."""
    w = W.WORKLOADS["dyntree60-v32000"]
    inp = W.make_inputs_np(w, seed=4, batch=12)
    parents = inp["parents"].copy()
    parents[5, 7] = 7                                 # node 7 its own parent
    for mode in (oracle.MODE_RESISPEC, oracle.MODE_SPECINFER):
        batched = oracle.verify(inp["target"], inp["draft"], parents, inp["cand"], 1.0, 21,
                                mode=mode, max_depth=6, want_dist=True)
        for b in range(12):
            one = oracle.verify(inp["target"][b:b + 1], inp["draft"][b:b + 1], parents[b],
                                inp["cand"][b:b + 1], 1.0, 21, mode=mode, max_depth=6,
                                seq_ids=np.array([b], np.int32), want_dist=True)
            for k in ("tokens", "accept_len", "nodes", "rejects", "status", "dist"):
                np.testing.assert_array_equal(batched[k][b], one[k][0])
        assert batched["status"][5] == oracle.ERR_TREE
        assert (np.delete(batched["status"], 5) & ~oracle.INFO_DEGENERATE == 0).all()


def test_random_trees_are_valid_and_candidates_come_from_parent_rows():
    rng = np.random.default_rng(0)
    trees = W.tree_random(rng, 40, 60, 6)
    for t in trees:
        assert ((t >= -1) & (t < np.arange(60))).all()
        assert W.tree_depth(t) <= 6
    # candidates drawn at a tiny temperature are the argmax of the parent's
    # draft row; every row has a distinct argmax, so each candidate names
    # its parent's row
    B, N, V = 40, 60, 400
    draft = rng.normal(0, 1, (B, N + 1, V)).astype(np.float32)
    for b in range(B):
        for r in range(N + 1):
            draft[b, r, r] = 50.0
    cand = W.candidates_np(rng, draft, trees, 1e-3)
    np.testing.assert_array_equal(cand, trees + 1)


@pytest.mark.parametrize("fill", [0, 1])
def test_oracle_denominator_update_matches_enumerator(fill):
    """Proxy-as-denominator variant (the test denominator becomes each
    rejection's proxy K): oracle draws against the independently enumerated
    law of the same rule, GetProxy invariants at every rejection, and the law
    differs from Algorithm 1's.  Also with the level fill."""
    V, k, n = 8, 3, 400_000
    zt, zd = _pq(43, V, scale=1.5, rho=0.3)
    target, draft, cand = _single_position_draws(6, V, k, n, zt, zd)
    out = oracle.verify(target, draft, W.tree_single(k), cand, 1.0, seed=4321,
                        mode=oracle.MODE_RESISPEC, seq_stride=0, check_invariants=True,
                        denom_update=True, fill=fill)
    assert (out["status"] & ~oracle.INFO_DEGENERATE == 0).all()
    assert out["inv_err"].max() < 1e-12
    p = sp_softmax(zt.astype(np.float64))
    q = sp_softmax(zd.astype(np.float64))
    dist, acc = en.single_position(p, q, k, oracle.MODE_RESISPEC, denom_update=True, fill=fill)
    pv, nb = chisq_pvalue(np.bincount(out["tokens"][:, 0], minlength=V), dist)
    assert pv > 1e-4, (pv, nb)
    which = np.where(out["accept_len"] > 0, out["nodes"][:, 0], k)
    pv2, _ = chisq_pvalue(np.bincount(which, minlength=k + 1), np.append(acc, 1 - acc.sum()))
    assert pv2 > 1e-4
    dist0, _ = en.single_position(p, q, k, oracle.MODE_RESISPEC, fill=fill)
    assert np.abs(dist - dist0).max() > 1e-3


def test_denominator_update_is_algorithm1_at_two_tokens():
    """V = 2: after a rejection the residual is the point mass on the other
    token under either denominator, so every later test of it accepts and
    every test of the rejected token rejects: the variant's outputs equal
    Algorithm 1's."""
    rng = np.random.default_rng(9)
    for _ in range(20):
        zt = rng.normal(0, 1.5, (1, 5, 2)).astype(np.float32)
        zd = rng.normal(0, 1.5, (1, 5, 2)).astype(np.float32)
        cand = rng.integers(0, 2, (300, 4)).astype(np.int32)
        kw = dict(mode=oracle.MODE_RESISPEC, seq_stride=0, want_dist=True)
        a = oracle.verify(zt[0], zd[0], W.tree_single(4), cand, 1.0, 3, **kw)
        b = oracle.verify(zt[0], zd[0], W.tree_single(4), cand, 1.0, 3, denom_update=True, **kw)
        for key in ("tokens", "accept_len", "nodes", "rejects", "dist"):
            np.testing.assert_array_equal(a[key], b[key])


def test_oracle_drafted_candidates_follow_q():
    """Drafting (Algorithm 1's x_1..x_k ~ Q i.i.d.): every drafted child of
    the root is a draw from the root's tempered draft softmax; the first two
    children are drawn independently of each other."""
    V, k, n = 16, 3, 200_000
    zt, zd = _pq(44, V, scale=1.5, rho=0.5)
    target = np.ascontiguousarray(np.broadcast_to(zt, (k + 1, V)), dtype=np.float32)
    draft = np.ascontiguousarray(np.broadcast_to(zd, (k + 1, V)), dtype=np.float32)
    cand = np.zeros((n, k), np.int32)
    out = oracle.verify(target, draft, W.tree_single(k), cand, 1.0, seed=77, seq_stride=0,
                        draft_children=True)
    q = sp_softmax(zd.astype(np.float64))
    d = out["drafted"]
    for j in range(k):
        assert (d[:, j] >= 0).all()
        assert chisq_pvalue(np.bincount(d[:, j], minlength=V), q)[0] > 1e-4
    joint = np.bincount(d[:, 0] * V + d[:, 1], minlength=V * V)
    assert chisq_pvalue(joint, np.outer(q, q).ravel())[0] > 1e-4
    # an accepted candidate is emitted as drafted
    acc = out["accept_len"] >= 1
    np.testing.assert_array_equal(out["tokens"][acc, 0], d[acc, out["nodes"][acc, 0]])


# ------------------------------------------------------------ fp32 error bound of proxy chains


def _fp32_softmax(z, T):
    """Tempered softmax as an fp32 evaluation: a = fp32(z c - M) (one
    rounding, as a fused multiply-add), 2^a in fp32, fp32 sum and divide."""
    c = np.float32(1.4426950408889634 / np.float32(T))
    z = z.astype(np.float32)
    M = np.float32(z.max() * c)
    a = (z.astype(np.float64) * np.float64(c) - np.float64(M)).astype(np.float32)
    e = np.exp2(a).astype(np.float32)
    return (e / e.sum(dtype=np.float32)).astype(np.float32)


def _fp32_proxy_chain(zt, zd, xs, fill):
    """The proxy-denominator chain of rejections of xs in fp32 arithmetic:
    the level is solved exactly on the fp32 values, every elementwise step
    is rounded to fp32."""
    f = np.float32
    R, D = _fp32_softmax(zt, 1.0), _fp32_softmax(zd, 1.0)
    rejected = []
    for x0 in xs:
        Z = f(D[x0] - R[x0])
        if not Z > 0:
            continue
        off = np.ones(R.size, bool)
        off[x0] = False
        off[rejected] = False
        R64, D64 = R.astype(np.float64), D.astype(np.float64)
        lam = Z
        if fill:
            lam = en.level_by_bisection(np.where(off, R64, 0.0), D64, x0, float(Z))
        if np.isfinite(lam):
            m = np.minimum((f(lam) * D).astype(f), R)
        else:
            m = np.where(D > 0, R, f(0))
        m = np.where(off, m, f(0))
        t = np.where(off, (R - m).astype(f), f(0))
        mu = f(0)
        if not fill or not np.isfinite(lam):
            mu = f(min(max((Z - m.sum(dtype=f)) / t.sum(dtype=f), 0), 1)) if t.sum() > 0 else f(0)
        r = (m + mu * t).astype(f)
        K = ((f(1) - mu) * t).astype(f)
        K[x0] = D[x0]       # K = R - r = 0 at the earlier rejected tokens
        R = (r / r.sum(dtype=f)).astype(f)
        D = K
        rejected.append(x0)
    return R.astype(np.float64)


@pytest.mark.parametrize("fill", [0, 1])
def test_proxy_chain_error_bound_covers_fp32(fill):
    """Reading R11: the oracle's per-token error bound of a proxy-denominator
    row covers an fp32 evaluation of the same rejections, token by token,
    on rows built to put tokens next to the level (R close to lam D), where
    the proxy K = R - r cancels."""
    rng = np.random.default_rng(31 + fill)
    V, k = 1500, 4
    worst_ratio, rows = 0.0, 0
    for trial in range(40):
        zt = rng.normal(0, 2.0, V).astype(np.float32)
        zd = (0.7 * zt + 0.7 * rng.normal(0, 2.0, V)).astype(np.float32)
        xs = list(rng.choice(V, size=k, p=sp_softmax(zd.astype(np.float64))))
        if trial % 3 == 0:
            xs[1] = xs[0]   # a duplicate rejection
        zt[xs] = -np.inf    # candidates the target excludes: every test rejects
        cand = np.asarray([xs], np.int32)
        target = np.broadcast_to(zt, (k + 1, V)).copy()
        draft = np.broadcast_to(zd, (k + 1, V)).copy()
        o = oracle.verify(target, draft, W.tree_single(k), cand, 1.0, 5, seq_stride=0,
                          want_dist=True, denom_update=True, fill=fill, want_dist_err=True,
                          decide_fp64=True)
        if o["accept_len"][0] != 0 or o["rejects"][0] != k:
            continue
        g = _fp32_proxy_chain(zt, zd, xs, fill)
        diff = np.abs(g - o["dist"][0])
        bound = o["dist_err"][0]
        assert (diff <= bound + 1e-12).all(), (trial, diff.max(), bound[np.argmax(diff - bound)])
        worst_ratio = max(worst_ratio, (diff / np.maximum(bound, 1e-300)).max())
        rows += 1
    assert rows >= 30
    assert worst_ratio > 1e-2   # the bound is not vacuous on these rows


def test_dist_err_is_zero_without_the_proxy_denominator():
    V, k = 300, 3
    rng = np.random.default_rng(4)
    zt = rng.normal(0, 2, (k + 1, V)).astype(np.float32)
    zd = rng.normal(0, 2, (k + 1, V)).astype(np.float32)
    cand = rng.integers(0, V, (8, k)).astype(np.int32)
    o = oracle.verify(zt, zd, W.tree_single(k), cand, 1.0, 5, seq_stride=0, want_dist=True,
                      fill=1, want_dist_err=True)
    assert (o["dist_err"] == 0).all()


@pytest.mark.parametrize("fill", [0, 1])
def test_oracle_z_applied_matches_enumerator(fill):
    """The Z_applied budget (Sec. 5.3 heuristic, reading R7): oracle draws
    against the law the enumerator derives with its own budget rule.  (By
    Theorem 2 every budget up to Z* reaches the ideal proxy, so this law is
    close to Algorithm 1's; the budgets themselves are compared below.)"""
    V, k, n = 8, 3, 400_000
    zt, zd = _pq(45, V, scale=1.5, rho=0.4)
    target, draft, cand = _single_position_draws(7, V, k, n, zt, zd)
    out = oracle.verify(target, draft, W.tree_single(k), cand, 1.0, seed=2468,
                        mode=oracle.MODE_RESISPEC, seq_stride=0, z_rule=1, fill=fill)
    assert (out["status"] & ~oracle.INFO_DEGENERATE == 0).all()
    p = sp_softmax(zt.astype(np.float64))
    q = sp_softmax(zd.astype(np.float64))
    dist, acc = en.single_position(p, q, k, oracle.MODE_RESISPEC, fill=fill, z_rule=1)
    pv, nb = chisq_pvalue(np.bincount(out["tokens"][:, 0], minlength=V), dist)
    assert pv > 1e-4, (pv, nb)
    which = np.where(out["accept_len"] > 0, out["nodes"][:, 0], k)
    pv2, _ = chisq_pvalue(np.bincount(which, minlength=k + 1), np.append(acc, 1 - acc.sum()))
    assert pv2 > 1e-4


def test_z_applied_budget_matches_enumerator():
    """The oracle's Z_applied budget against the enumerator's own, on rows
    where the capacity bound Z* exceeds the gap (the heuristic's case) and
    where it does not."""
    rng = np.random.default_rng(46)
    above = 0
    for _ in range(300):
        V = int(rng.integers(2, 30))
        R = rng.dirichlet(np.full(V, 3.0))
        q = rng.dirichlet(np.full(V, 3.0))
        x0 = int(np.argmax(q - R))
        if not q[x0] > R[x0]:
            continue
        zo, ze = oracle.budget(R, q, x0, z_rule=1), en.budget(R, q, x0, z_rule=1)
        assert zo == pytest.approx(ze, rel=1e-14, abs=1e-16)
        assert oracle.budget(R, q, x0) == pytest.approx(en.budget(R, q, x0), abs=1e-16)
        above += zo > q[x0] - R[x0] + 1e-12
    assert above > 30
