"""GPU parity: the CUDA verification path against the fp64 oracle on the
same seeded inputs, through the C ABI (see tests/parity.py for the rule)."""
import dataclasses
import functools

import numpy as np
import pytest
from scipy.special import softmax as sp_softmax

import oracle
import paper_2608_24411_gb300 as rs
from oracle import enumerator as en
from paper_2608_24411_gb300 import workloads as W
from tests import parity as P
from tests.test_oracle_walk import chisq_pvalue

pytestmark = pytest.mark.gpu
MODES = [rs.MODE_RESISPEC, rs.MODE_SPECINFER]
KERNELS = ["resident", "stream"]


@pytest.fixture(scope="module", autouse=True)
def built():
    rs.build()
    rs.load_library()


@functools.lru_cache(maxsize=2)
def _inputs(name, seed, batch):
    """make_inputs_np for a named workload, kept for the next test with the
    same inputs (parametrized tests run next to each other); callers must
    not modify the arrays."""
    return W.make_inputs_np(W.WORKLOADS[name], seed=seed, batch=batch)


def _np_inputs_to_gpu(inp):
    import torch
    return (P.to_device(inp["target"]), P.to_device(inp["draft"]),
            torch.as_tensor(inp["parents"], dtype=torch.int32, device="cuda"),
            torch.as_tensor(inp["cand"], dtype=torch.int32, device="cuda"))


def _refused_on_resident(zt, zd, pa, ca, T, seed, D, **kw):
    """SpecInfer runs on the streaming kernel only: forcing the resident
    kernel is an argument error, returned before any launch."""
    with pytest.raises(rs.ResispecError) as e:
        P.run_gpu(zt, zd, pa, ca, T, seed, D, mode=rs.MODE_SPECINFER, kernel="resident", **kw)
    assert e.value.code == rs.E_ARG


def _check(inp, mode, seed, **kw):
    zt, zd, pa, ca = _np_inputs_to_gpu(inp)
    D = int(inp["max_depth"])
    if mode == rs.MODE_SPECINFER and kw.get("kernel") == "resident":
        _refused_on_resident(zt, zd, pa, ca, inp["temperature"], seed, D,
                             **{k: v for k, v in kw.items() if k != "kernel"})
        return None, None
    g = P.run_gpu(zt, zd, pa, ca, inp["temperature"], seed, D, mode=mode, **kw)
    o = P.run_oracle(inp["target"], inp["draft"], inp["parents"], inp["cand"],
                     inp["temperature"], seed, D, mode, z_rule=kw.get("z_rule", 0),
                     denom_update=kw.get("proxy_denominator", False), fill=kw.get("fill", 0))
    rep = P.compare(g, o)
    n, near = rep["sequences"], rep["mismatch_in_ties"]
    # near-tie differences are allowed but must stay rare
    assert near <= max(2, 0.002 * n), (near, n)
    assert g["status"][0] & ~rs.INFO_DEGENERATE == 0
    return g, o


@pytest.mark.parametrize("mode", MODES)
@pytest.mark.parametrize("dtype", ["f32", "bf16"])
@pytest.mark.parametrize("cluster,threads", [(0, 0), (1, 256), (1, 512), (16, 256)])
def test_parity_max_vocab(cluster, threads, dtype, mode):
    """The largest vocabulary (V = 262144): the automatic launch shape, one
    CTA per sequence (a slice of 128 chunks at 256 threads, the search's
    chunk-total limit, without chunk records), and clusters of 16; a chain
    of depth 4 with 3 candidates per level, zipf logits."""
    _check(_max_vocab_inputs(dtype), mode, seed=410 + cluster, cluster_size=cluster,
           block_threads=threads, kernel="stream")


@functools.lru_cache(maxsize=2)
def _max_vocab_inputs(dtype):
    w = dataclasses.replace(W.WORKLOADS["tiny-chain-v64"], vocab=rs.MAX_VOCAB, dtype=dtype,
                            gen="zipf", scale=3.0, slope=1.1, name="tiny-chain-vmax")
    return W.make_inputs_np(w, seed=41, batch=8)


def test_device_philox_matches_numpy():
    import torch
    from tests.test_oracle_pins import _np_philox_block
    rng = np.random.default_rng(0)
    n = 4000
    seq = rng.integers(0, 1 << 31, n).astype(np.int32)
    row = rng.integers(0, 1 << 31, n).astype(np.int32)
    for seed in (0, 1, 2 ** 64 - 1, 0x123456789ABCDEF0):
        u0, u1 = rs.uniforms(seed, torch.as_tensor(seq, device="cuda"),
                             torch.as_tensor(row, device="cuda"))
        u0, u1 = u0.cpu().numpy(), u1.cpu().numpy()
        for i in range(0, n, 97):
            blk = _np_philox_block([int(row[i]), int(seq[i]), 0, 0], [seed, 0])
            assert u0[i] == np.float32((int(blk[0]) >> 40) / 2.0 ** 24)
            assert u1[i] == np.float32((int(blk[1]) >> 40) / 2.0 ** 24)


@pytest.mark.parametrize("kernel", KERNELS)
@pytest.mark.parametrize("mode", MODES)
@pytest.mark.parametrize("cluster", [0, 1, 16])
def test_parity_tiny_chain_10000(mode, cluster, kernel):
    """Chain depth 4 with k = 3, V = 64, fp32: 10,000 independent problems
    from seed 0 (10,000 verify steps) in one batch."""
    w = W.WORKLOADS["tiny-chain-v64"]
    inp = W.make_inputs_np(w, seed=0, batch=10_000)
    _check(inp, mode, seed=0, cluster_size=cluster, kernel=kernel)


@pytest.mark.parametrize("kernel", KERNELS)
@pytest.mark.parametrize("mode", MODES)
def test_parity_tree60_v32000(mode, kernel):
    w = W.WORKLOADS["tree60-v32000"]
    inp = _inputs(w.name, 1, 256)
    _check(inp, mode, seed=11, kernel=kernel)


@pytest.mark.parametrize("kernel", KERNELS)
def test_parity_tree60_v32000_per_call_seeds(kernel):
    """Batch 1, one call per step with seed = base + step (the paper's seed
    schedule), launch shape chosen automatically for a single sequence."""
    w = W.WORKLOADS["tree60-v32000"]
    for step in range(12):
        inp = W.make_inputs_np(w, seed=100 + step, batch=1)
        _check(inp, rs.MODE_RESISPEC, seed=5000 + step, kernel=kernel)


@pytest.mark.parametrize("kernel", KERNELS)
@pytest.mark.parametrize("mode", MODES)
def test_parity_chain8x4_v128256(mode, kernel):
    w = W.WORKLOADS["chain8x4-v128256-b16"]
    for step in range(3):
        inp = W.make_inputs_np(w, seed=20 + step, batch=16)
        _check(inp, mode, seed=900 + step, kernel=kernel)


@pytest.mark.parametrize("kernel", KERNELS)
@pytest.mark.parametrize("V", [1, 2, 3, 7, 61, 999, 1000, 1003, 4104, 20000, 20001])
@pytest.mark.parametrize("dtype", ["f32", "bf16"])
@pytest.mark.parametrize("no_tma", [False, True])
def test_parity_ragged_vocab(V, dtype, no_tma, kernel):
    """Vocabularies that leave ragged slice tails, empty CTAs (V < cluster
    slices), slices of several streaming chunks with a ragged last chunk,
    and rows that are not 16-byte aligned (plain-load path)."""
    base = W.Workload(name="ragged", batch=64, vocab=V, dtype=dtype, gen="gauss", scale=2.0,
                      slope=0.0, rho=0.6, temperature=0.9, tree=("levels", (3, 2, 1)), steps=1)
    inp = W.make_inputs_np(base, seed=V, batch=64)
    for cluster in (0, 1, 4, 11, 16):
        if kernel == "resident" and cluster == 1 and V > 4104:
            continue  # two fp32 rows of V = 20001 do not fit one CTA's shared memory
        for mode in MODES:
            _check(inp, mode, seed=V + cluster, cluster_size=cluster, no_tma=no_tma,
                   kernel=kernel)


@pytest.mark.parametrize("kernel", KERNELS)
@pytest.mark.parametrize("threads", [256, 512])
def test_launch_shapes_agree(threads, kernel):
    w = W.WORKLOADS["tree60-v32000"]
    inp = W.make_inputs_np(w, seed=2, batch=64)
    ref = None
    # one CTA cannot hold two V = 32000 fp32 rows (resident kernel)
    clusters = (2, 3, 4, 8, 12, 16) if kernel == "resident" else (1, 2, 3, 5, 8, 16)
    for cluster in clusters:
        g, o = _check(inp, rs.MODE_RESISPEC, seed=3, cluster_size=cluster, block_threads=threads,
                      kernel=kernel)
        clean = (o["accept_margin"] > P.ACCEPT_TIE) & (o["sample_margin"] > P.SAMPLE_TIE)
        if ref is not None:
            assert (g["tokens"][clean] == ref[clean]).all()
        ref = g["tokens"]


def test_kernels_agree_away_from_ties():
    """Both kernels on the same inputs: identical outputs wherever the
    oracle sees no near tie."""
    w = W.WORKLOADS["chain8x4-v128256-b16"]
    inp = W.make_inputs_np(w, seed=7, batch=16)
    g1, o = _check(inp, rs.MODE_RESISPEC, seed=70, kernel="resident")
    g2, _ = _check(inp, rs.MODE_RESISPEC, seed=70, kernel="stream")
    clean = (o["accept_margin"] > P.ACCEPT_TIE) & (o["sample_margin"] > P.SAMPLE_TIE)
    assert (g1["tokens"][clean] == g2["tokens"][clean]).all()
    assert (g1["accept_len"][clean] == g2["accept_len"][clean]).all()


@pytest.mark.parametrize("kernel", KERNELS)
def test_repeat_runs_bit_identical(kernel):
    w = W.WORKLOADS["chain8x4-v128256-b16"]
    inp = W.make_inputs_np(w, seed=5, batch=16)
    zt, zd, pa, ca = _np_inputs_to_gpu(inp)
    a = P.run_gpu(zt, zd, pa, ca, inp["temperature"], 77, inp["max_depth"], kernel=kernel)
    b = P.run_gpu(zt, zd, pa, ca, inp["temperature"], 77, inp["max_depth"], kernel=kernel)
    for k in ("tokens", "accept_len", "nodes", "rejects", "dist"):
        np.testing.assert_array_equal(a[k], b[k])


@pytest.mark.parametrize("mode", MODES)
def test_wide_fanout(mode):
    """A star of MAX_FANOUT_STREAM children (the streaming kernel's limit)
    whose candidates the target all but excludes (target logit -30 at every
    candidate: every test rejects, the walk reaches the last child, 128
    residual maps) on both kernels; one child more: the streaming kernel
    reports ERR_FANOUT when the walk reaches the 129th child, the resident
    kernel verifies (ResiSpec; SpecInfer runs on the streaming kernel only)."""
    import torch
    V = 3000
    for kids in (rs.MAX_FANOUT_STREAM, rs.MAX_FANOUT_STREAM + 1):
        parents = np.full(kids, -1, np.int32)
        rng = np.random.default_rng(kids)
        zt = rng.normal(0, 2, (8, kids + 1, V)).astype(np.float32)
        zd = rng.normal(0, 2, (8, kids + 1, V)).astype(np.float32)
        cand = rng.integers(0, V, (8, kids)).astype(np.int32)
        for b in range(8):
            zt[b, 0, cand[b]] = -30.0
        inp = {"target": zt, "draft": zd, "parents": parents, "cand": cand, "temperature": 1.0,
               "max_depth": 1}
        _check(inp, mode, seed=kids, kernel="resident")
        if kids <= rs.MAX_FANOUT_STREAM:
            _check(inp, mode, seed=kids, kernel="stream")
        else:
            # SpecInfer rejects every candidate, so the walk reaches the
            # 129th child; ResiSpec's shaped residual moves toward q and
            # accepts a later candidate first (the method's over-acceptance)
            zt_, zd_, pa, ca = _np_inputs_to_gpu(inp)
            g = P.run_gpu(zt_, zd_, pa, ca, 1.0, kids, 1, mode=mode, kernel="stream")
            o = P.run_oracle(zt, zd, parents, cand, 1.0, kids, 1, mode)
            far = o["rejects"] >= rs.MAX_FANOUT_STREAM
            assert far.any() == (mode == rs.MODE_SPECINFER)
            assert (g["accept_len"][far] == -1).all()
            assert (g["status"][0] & rs.ERR_FANOUT) == (rs.ERR_FANOUT if far.any() else 0)
            clean = ~far & (o["accept_margin"] > P.ACCEPT_TIE) & (o["sample_margin"] > P.SAMPLE_TIE)
            assert (g["accept_len"][clean] == o["accept_len"][clean]).all()
            assert (g["tokens"][clean] == o["tokens"][clean]).all()


@pytest.mark.parametrize("kernel", KERNELS)
def test_empty_tree_and_empty_batch(kernel):
    import torch
    V = 5000
    rng = np.random.default_rng(4)
    zt = rng.normal(0, 3, (40, 1, V)).astype(np.float32)
    pa = np.zeros(0, np.int32)
    ca = np.zeros((40, 0), np.int32)
    g = P.run_gpu(P.to_device(zt), P.to_device(zt), torch.zeros(0, dtype=torch.int32, device="cuda"),
                  torch.zeros((40, 0), dtype=torch.int32, device="cuda"), 1.0, 8, 0,
                  kernel=kernel)
    o = P.run_oracle(zt, zt, pa, ca, 1.0, 8, 0, rs.MODE_RESISPEC)
    P.compare(g, o)
    assert (g["accept_len"] == 0).all()
    e = torch.zeros((0, 1, V), device="cuda")
    toks, alen = rs.verify(e, e, torch.zeros(0, dtype=torch.int32, device="cuda"),
                           torch.zeros((0, 0), dtype=torch.int32, device="cuda"), 1.0, 0,
                           max_depth=0)
    assert toks.shape == (0, 1) and alen.shape == (0,)


@pytest.mark.parametrize("kernel", KERNELS)
def test_shared_rows_seq_stride_zero(kernel):
    import torch
    w = W.WORKLOADS["tiny-chain-v64"]
    inp = W.make_inputs_np(w, seed=3, batch=1)
    B = 3000
    rng = np.random.default_rng(3)
    cand = rng.integers(0, 64, (B, w.num_nodes)).astype(np.int32)
    zt = P.to_device(inp["target"][0])
    zd = P.to_device(inp["draft"][0])
    pa = torch.as_tensor(inp["parents"], device="cuda")
    g = P.run_gpu(zt, zd, pa, torch.as_tensor(cand, device="cuda"), 1.0, 6, w.max_depth,
                  seq_stride=0, kernel=kernel)
    o = P.run_oracle(inp["target"][0], inp["draft"][0], inp["parents"], cand, 1.0, 6,
                     w.max_depth, rs.MODE_RESISPEC, seq_stride=0)
    P.compare(g, o)


@pytest.mark.parametrize("kernel", KERNELS)
def test_error_contract_matches_oracle(kernel):
    import torch
    parents = W.tree_levels([2, 2])
    V, B = 1024, 9
    rng = np.random.default_rng(1)
    zt = rng.normal(0, 1, (B, 7, V)).astype(np.float32)
    zd = zt.copy()
    cand = rng.integers(0, V, (B, 6)).astype(np.int32)
    cand[1, 0] = V
    cand[5, 0] = -3
    zt[2, 0, 3] = np.nan
    zt[3, 0, :] = -np.inf
    zt[4, 6, 0] = np.nan              # never visited
    zd[6, 0, 100] = np.inf
    zt[8, 0, :] = -np.inf             # NaN hidden among -inf logits
    zt[8, 0, 517] = np.nan
    g = P.run_gpu(P.to_device(zt), P.to_device(zd), torch.as_tensor(parents, device="cuda"),
                  torch.as_tensor(cand, device="cuda"), 1.0, 0, 2, want_dist=False,
                  kernel=kernel)
    o = P.run_oracle(zt, zd, parents, cand, 1.0, 0, 2, rs.MODE_RESISPEC, want_dist=False)
    np.testing.assert_array_equal(g["accept_len"] == -1, o["accept_len"] == -1)
    assert list(np.nonzero(o["accept_len"] == -1)[0]) == [1, 2, 3, 5, 6, 8]
    assert o["status"][8] == oracle.ERR_NONFINITE
    assert (g["tokens"][[1, 2, 3, 5, 6, 8]] == -1).all()
    want = int(np.bitwise_or.reduce(o["status"]))
    assert g["status"][0] & ~rs.INFO_DEGENERATE == want & ~oracle.INFO_DEGENERATE
    # depth overflow and a tree that is not in topological order
    g = P.run_gpu(P.to_device(zt[:1]), P.to_device(zd[:1]), torch.as_tensor(parents, device="cuda"),
                  torch.as_tensor(cand[:1], device="cuda"), 1.0, 0, 1, want_dist=False,
                  kernel=kernel)
    assert g["accept_len"][0] == -1 and g["status"][0] == rs.ERR_DEPTH
    bad = torch.as_tensor(np.array([-1, 1, 0, 0, 1, 1], np.int32), device="cuda")
    g = P.run_gpu(P.to_device(zt[:2]), P.to_device(zd[:2]), bad,
                  torch.as_tensor(cand[:2], device="cuda"), 1.0, 0, 3, want_dist=False,
                  kernel=kernel)
    assert (g["accept_len"] == -1).all() and g["status"][0] == rs.ERR_TREE


def test_synchronous_errors_on_device():
    import torch
    t = torch.zeros((1, 2, 8), device="cuda")
    pa = torch.zeros(1, dtype=torch.int32, device="cuda") - 1
    ca = torch.zeros((1, 1), dtype=torch.int32, device="cuda")
    with pytest.raises(rs.ResispecError):
        rs.verify(t, t, pa, ca, 0.0, 0, max_depth=1)
    with pytest.raises(rs.ResispecError):
        rs.verify(t, t, pa, ca, 1.0, 0, max_depth=1, cluster_size=17)


def test_nondefault_stream():
    import torch
    w = W.WORKLOADS["tree60-v32000"]
    inp = W.make_inputs_np(w, seed=9, batch=32)
    zt, zd, pa, ca = _np_inputs_to_gpu(inp)
    s = torch.cuda.Stream()
    s.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(s):
        toks, alen = rs.verify(zt, zd, pa, ca, 1.0, 4, max_depth=inp["max_depth"])
    s.synchronize()
    o = P.run_oracle(inp["target"], inp["draft"], inp["parents"], inp["cand"], 1.0, 4,
                     inp["max_depth"], rs.MODE_RESISPEC, want_dist=False)
    P.compare({"tokens": toks.cpu().numpy(), "accept_len": alen.cpu().numpy()}, o,
              check_dist=False)


# ------------------------------------------------------------ full-size workloads


def _sampled_parity(w, seed, call_seed, rows, mode=rs.MODE_RESISPEC, batch=None, rho=None,
                    kernel=None, **kw):
    """Full-size inputs drawn on the GPU; the oracle recomputes the sampled
    sequences `rows` one by one from the same tensors."""
    import torch
    inp = W.make_inputs_torch(w, seed, "cuda", batch=batch, rho=rho)
    D = inp["max_depth"]
    if mode == rs.MODE_SPECINFER and kernel == "resident":
        _refused_on_resident(inp["target"], inp["draft"], inp["parents"], inp["cand"],
                             w.temperature, call_seed, D, **kw)
        return None
    g = P.run_gpu(inp["target"], inp["draft"], inp["parents"], inp["cand"], w.temperature,
                  call_seed, D, mode=mode, kernel=kernel, **kw)
    ridx = torch.as_tensor(rows, device="cuda")
    th = P.to_host_logits(inp["target"].index_select(0, ridx))
    dh = P.to_host_logits(inp["draft"].index_select(0, ridx))
    ch = inp["cand"].index_select(0, ridx).cpu().numpy()
    pa = inp["parents_np"][rows] if inp["parents_np"].ndim == 2 else inp["parents_np"]
    o = P.run_oracle(th, dh, pa, ch, w.temperature, call_seed, D, mode,
                     seq_ids=np.asarray(rows, np.int32), z_rule=kw.get("z_rule", 0),
                     denom_update=kw.get("proxy_denominator", False), fill=kw.get("fill", 0))
    rep = P.compare(g, o, rows=rows)
    assert rep["mismatch_in_ties"] <= 1, rep
    assert g["status"][0] & ~rs.INFO_DEGENERATE == 0
    assert (g["accept_len"] >= 0).all()
    del inp
    torch.cuda.empty_cache()
    return g


@pytest.mark.parametrize("kernel", [None, "resident"])
@pytest.mark.parametrize("rho", [0.5, 0.8, 0.95])
def test_parity_binary5_v151936_full_size(rho, kernel):
    """B = 64, V = 151936 fp32, full binary tree of depth 5, in the launch
    shape the benchmark times (kernel None: the automatic choice); 8 sampled
    sequences per call checked."""
    w = W.WORKLOADS["binary5-v151936-b64"]
    _sampled_parity(w, seed=31, call_seed=1000, rows=[0, 9, 17, 26, 35, 44, 53, 63], rho=rho,
                    kernel=kernel)


@pytest.mark.parametrize("kernel", KERNELS)
def test_parity_binary5_specinfer_full_size(kernel):
    w = W.WORKLOADS["binary5-v151936-b64"]
    _sampled_parity(w, seed=32, call_seed=1001, rows=[1, 20, 40, 62], mode=rs.MODE_SPECINFER,
                    kernel=kernel)


def _spread_rows(B, n):
    """n sequence indices spread over a batch of B (first and last included)."""
    return sorted({int(round(i * (B - 1) / (n - 1))) for i in range(n)})


@pytest.mark.parametrize("B", [32, 128])
@pytest.mark.parametrize("k", [2, 4, 8, 16])
def test_parity_single_position_v256000(k, B):
    """Single position with k candidates, V = 256000 bf16, at the batch and
    in the launch shape the benchmark times; 8 sampled sequences."""
    w = W.WORKLOADS[f"single-k{k}-v256000-b{B}"]
    _sampled_parity(w, seed=40 + k + B, call_seed=77 + k, rows=_spread_rows(B, 8))


@pytest.mark.parametrize("kernel", KERNELS)
def test_parity_single_position_v256000_kernels(kernel):
    w = W.WORKLOADS["single-k16-v256000-b32"]
    _sampled_parity(w, seed=45, call_seed=79, rows=[0, 7, 15, 31], kernel=kernel)


@pytest.mark.parametrize("B", [32, 128])
def test_parity_tree488_v256000(B):
    """Tree [8, 4, 2, 2, 1, 1] (488 nodes), V = 256000 bf16, the whole batch
    (B = 128: 64 GB of logits) in the launch shape the benchmark times;
    6 sampled sequences."""
    w = W.WORKLOADS[f"tree488-v256000-b{B}"]
    _sampled_parity(w, seed=50 + B, call_seed=78, rows=_spread_rows(B, 6))


@pytest.mark.parametrize("kernel", KERNELS)
def test_parity_tree488_v256000_kernels(kernel):
    w = W.WORKLOADS["tree488-v256000-b32"]
    _sampled_parity(w, seed=50, call_seed=78, rows=[0, 5], batch=6, kernel=kernel)


# ------------------------------------------------------------ exactness on the GPU


def test_gpu_specinfer_million_draws_v32000(kernel="stream"):
    """SpecInfer mode is distribution-exact: 1e6 GPU draws at V = 32000 (one
    shared set of rows, fresh candidates per draw) do not reject p."""
    import torch
    V, k, n = 32000, 4, 1_000_000
    w = W.WORKLOADS["tree60-v32000"]
    rng = np.random.default_rng(12)
    zt, zd = W.logits_np(rng, 1, V, "zipf", w.scale, w.slope, w.rho)
    zt_b, zd_b = W.f32_to_bf16_bits(zt[0]), W.f32_to_bf16_bits(zd[0])
    rows_t = np.ascontiguousarray(np.broadcast_to(zt_b, (k + 1, V)))
    rows_d = np.ascontiguousarray(np.broadcast_to(zd_b, (k + 1, V)))
    q = torch.softmax(torch.as_tensor(W.bf16_bits_to_f32(zd_b), dtype=torch.float64,
                                      device="cuda"), dim=0)
    gen = torch.Generator(device="cuda")
    gen.manual_seed(3)
    cand = torch.multinomial(q, n * k, replacement=True, generator=gen).to(torch.int32)
    cand = cand.view(n, k).contiguous()
    toks, alen = rs.verify(P.to_device(rows_t), P.to_device(rows_d),
                           torch.full((k,), -1, dtype=torch.int32, device="cuda"), cand, 1.0,
                           2024, max_depth=1, mode=rs.MODE_SPECINFER, seq_stride=0,
                           kernel=kernel)
    first = toks[:, 0].to(torch.int64)
    assert int(first.min()) >= 0
    counts = torch.bincount(first, minlength=V).cpu().numpy()
    p = sp_softmax(W.bf16_bits_to_f32(zt_b).astype(np.float64))
    pv, nb = chisq_pvalue(counts, p)
    assert pv > 1e-4, (pv, nb)


@pytest.mark.parametrize("kernel", KERNELS)
def test_gpu_resispec_million_draws_vs_enumerator(kernel):
    """ResiSpec mode on the GPU follows the enumerated law of Algorithm 1
    (and not p: the documented bias)."""
    import torch
    V, k, n = 16, 3, 1_000_000
    rng = np.random.default_rng(5)
    zt = (2.0 * rng.standard_normal(V)).astype(np.float32)
    zd = (0.8 * zt + 1.2 * rng.standard_normal(V)).astype(np.float32)
    p, q = sp_softmax(zt.astype(np.float64)), sp_softmax(zd.astype(np.float64))
    cand = rng.choice(V, size=(n, k), p=q).astype(np.int32)
    toks, _ = rs.verify(P.to_device(np.broadcast_to(zt, (k + 1, V)).copy()),
                        P.to_device(np.broadcast_to(zd, (k + 1, V)).copy()),
                        torch.full((k,), -1, dtype=torch.int32, device="cuda"),
                        torch.as_tensor(cand, device="cuda"), 1.0, 99, max_depth=1,
                        seq_stride=0, kernel=kernel)
    counts = np.bincount(toks[:, 0].cpu().numpy(), minlength=V)
    dist, _ = en.single_position(p, q, k, en.MODE_RESISPEC)
    assert chisq_pvalue(counts, dist)[0] > 1e-4
    assert chisq_pvalue(counts, p)[0] < 1e-12


@pytest.mark.parametrize("kernel", KERNELS)
@pytest.mark.parametrize("mode", MODES)
def test_parity_dynamic_trees(mode, kernel):
    """A random 60-node tree of depth <= 6 per sequence ([B, N] parents),
    64 sequences, V = 32000 bf16: every sequence against the oracle."""
    w = W.WORKLOADS["dyntree60-v32000"]
    inp = W.make_inputs_np(w, seed=61, batch=64)
    assert inp["parents"].shape == (64, 60)
    _check(inp, mode, seed=610 + mode, kernel=kernel)


@pytest.mark.parametrize("kernel", KERNELS)
def test_dynamic_tree_error_marks_only_its_sequence(kernel):
    w = W.WORKLOADS["dyntree60-v32000"]
    inp = W.make_inputs_np(w, seed=62, batch=16)
    inp["parents"] = inp["parents"].copy()
    inp["parents"][3, 10] = 11                        # a parent after its child
    zt, zd, pa, ca = _np_inputs_to_gpu(inp)
    g = P.run_gpu(zt, zd, pa, ca, inp["temperature"], 5, 6, kernel=kernel)
    o = P.run_oracle(inp["target"], inp["draft"], inp["parents"], inp["cand"],
                     inp["temperature"], 5, 6, rs.MODE_RESISPEC)
    assert g["accept_len"][3] == -1 and (g["tokens"][3] == -1).all()
    assert o["status"][3] == rs.ERR_TREE
    assert g["status"][0] & rs.ERR_TREE
    keep = np.arange(16) != 3
    clean = keep & (o["accept_margin"] > P.ACCEPT_TIE) & (o["sample_margin"] > P.SAMPLE_TIE)
    assert (g["accept_len"][clean] == o["accept_len"][clean]).all()
    assert (g["tokens"][clean] == o["tokens"][clean]).all()


@pytest.mark.parametrize("kernel", [None, "resident"])
def test_parity_dynamic_trees_v128256_full_size(kernel):
    """B = 64, V = 128256 bf16, a random 60-node tree per sequence, in the
    launch shape the benchmark times (kernel None); 8 sampled sequences."""
    w = W.WORKLOADS["dyntree60-v128256-b64"]
    _sampled_parity(w, seed=63, call_seed=1003, rows=[0, 9, 17, 26, 35, 44, 53, 63],
                    kernel=kernel)


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
@pytest.mark.parametrize("V", [8, 64, 1000, 20001])
def test_parity_z_applied_budget(V, dtype):
    """The Z_applied budget variant (max(Z*, gap) clamped to 1 - R(x0)) on
    close drafts (rho = 0.9, so min p / q can exceed the gap at a node's
    first rejection) with single-child levels (a rejected only child leads
    to a draw from the shaped residual, where the budget shows), every
    sequence against the oracle with the same rule; at small V the variant
    must change some walks."""
    base = W.Workload(name="zapp", batch=2000, vocab=V, dtype=dtype, gen="gauss", scale=1.0,
                      slope=0.0, rho=0.9, temperature=1.0, tree=("levels", (2, 1, 1)), steps=1)
    B = 2000 if V <= 1000 else 200
    inp = W.make_inputs_np(base, seed=V + 5, batch=B)
    g, o = _check(inp, rs.MODE_RESISPEC, seed=77, z_rule=rs.Z_RULE_APPLIED)
    o0 = P.run_oracle(inp["target"], inp["draft"], inp["parents"], inp["cand"],
                      inp["temperature"], 77, int(inp["max_depth"]), rs.MODE_RESISPEC, z_rule=0)
    if V <= 1000:
        assert (o0["tokens"] != o["tokens"]).any(axis=1).sum() > 0


def test_parity_z_applied_tree60():
    w = W.WORKLOADS["tree60-v32000"]
    inp = _inputs(w.name, 8, 256)
    _check(inp, rs.MODE_RESISPEC, seed=88, z_rule=rs.Z_RULE_APPLIED)


@pytest.mark.parametrize("wl", ["tree60-v32000", "chain8x4-v128256-b16", "dyntree60-v32000"])
def test_parity_proxy_denominator(wl):
    """The proxy-as-denominator variant (the paper's EAGLE integration): the
    accept tests and the next GetProxy use each rejection's proxy; every
    sequence against the oracle with the same rule, which must change some
    walks."""
    w = W.WORKLOADS[wl]
    inp = _inputs(w.name, 13, 256 if wl != "chain8x4-v128256-b16" else 16)
    g, o = _check(inp, rs.MODE_RESISPEC, seed=131, proxy_denominator=True)
    o0 = P.run_oracle(inp["target"], inp["draft"], inp["parents"], inp["cand"],
                      inp["temperature"], 131, int(inp["max_depth"]), rs.MODE_RESISPEC)
    if wl != "chain8x4-v128256-b16":
        assert ((o0["tokens"] != o["tokens"]).any(axis=1) | (o0["rejects"] != o["rejects"])).any()


@pytest.mark.parametrize("mode", MODES)
def test_proxy_denominator_wide_fanout(mode):
    """128 children whose candidates the target all but excludes: up to 128
    proxy updates at one node, against the oracle (SpecInfer: the flag has
    no effect)."""
    V, kids = 3000, rs.MAX_FANOUT_STREAM
    rng = np.random.default_rng(kids)
    zt = rng.normal(0, 2, (8, kids + 1, V)).astype(np.float32)
    zd = rng.normal(0, 2, (8, kids + 1, V)).astype(np.float32)
    cand = rng.integers(0, V, (8, kids)).astype(np.int32)
    for b in range(8):
        zt[b, 0, cand[b]] = -30.0
    inp = {"target": zt, "draft": zd, "parents": np.full(kids, -1, np.int32), "cand": cand,
           "temperature": 1.0, "max_depth": 1}
    _check(inp, mode, seed=kids, proxy_denominator=True)


def test_parity_proxy_denominator_binary5_full_size():
    w = W.WORKLOADS["binary5-v151936-b64"]
    _sampled_parity(w, seed=33, call_seed=1004, rows=[2, 19, 37, 58], proxy_denominator=True)


def test_gpu_proxy_denominator_million_draws_vs_enumerator():
    """The proxy-as-denominator variant on the GPU follows its own
    enumerated law."""
    import torch
    V, k, n = 16, 3, 1_000_000
    rng = np.random.default_rng(6)
    zt = (2.0 * rng.standard_normal(V)).astype(np.float32)
    zd = (0.8 * zt + 1.2 * rng.standard_normal(V)).astype(np.float32)
    p, q = sp_softmax(zt.astype(np.float64)), sp_softmax(zd.astype(np.float64))
    cand = rng.choice(V, size=(n, k), p=q).astype(np.int32)
    toks, _ = rs.verify(P.to_device(np.broadcast_to(zt, (k + 1, V)).copy()),
                        P.to_device(np.broadcast_to(zd, (k + 1, V)).copy()),
                        torch.full((k,), -1, dtype=torch.int32, device="cuda"),
                        torch.as_tensor(cand, device="cuda"), 1.0, 98, max_depth=1,
                        seq_stride=0, proxy_denominator=True)
    counts = np.bincount(toks[:, 0].cpu().numpy(), minlength=V)
    dist, _ = en.single_position(p, q, k, en.MODE_RESISPEC, denom_update=True)
    dist0, _ = en.single_position(p, q, k, en.MODE_RESISPEC)
    assert chisq_pvalue(counts, dist)[0] > 1e-4
    assert np.abs(dist - dist0).max() > 1e-3


# ------------------------------------------------------------ level fill


@pytest.mark.parametrize("wl", ["tree60-v32000", "chain8x4-v128256-b16", "dyntree60-v32000"])
def test_parity_level_fill(wl):
    """GetProxy's deficit raised to a level (r = min(lam q, R) with sum r =
    Z): every sequence against the oracle's exact level, which must change
    some walks against the default fill."""
    w = W.WORKLOADS[wl]
    inp = _inputs(w.name, 17, 256 if wl != "chain8x4-v128256-b16" else 16)
    g, o = _check(inp, rs.MODE_RESISPEC, seed=171, fill=rs.FILL_LEVEL)
    o0 = P.run_oracle(inp["target"], inp["draft"], inp["parents"], inp["cand"],
                      inp["temperature"], 171, int(inp["max_depth"]), rs.MODE_RESISPEC)
    if wl != "chain8x4-v128256-b16":
        assert ((o0["tokens"] != o["tokens"]).any(axis=1) | (o0["rejects"] != o["rejects"])).any()


@pytest.mark.parametrize("other", [dict(proxy_denominator=True), dict(z_rule=rs.Z_RULE_APPLIED)])
def test_parity_level_fill_with_other_variants(other):
    """The level fill combined with the proxy denominator (the level is
    taken against the current denominator) and with the Z_applied budget."""
    w = W.WORKLOADS["tree60-v32000"]
    inp = _inputs(w.name, 19, 256)
    _check(inp, rs.MODE_RESISPEC, seed=191, fill=rs.FILL_LEVEL, **other)


@pytest.mark.parametrize("mode", MODES)
def test_level_fill_wide_fanout(mode):
    """128 children whose candidates the target all but excludes: up to 128
    level searches at one node (SpecInfer: the flag has no effect)."""
    V, kids = 3000, rs.MAX_FANOUT_STREAM
    rng = np.random.default_rng(kids + 1)
    zt = rng.normal(0, 2, (8, kids + 1, V)).astype(np.float32)
    zd = rng.normal(0, 2, (8, kids + 1, V)).astype(np.float32)
    cand = rng.integers(0, V, (8, kids)).astype(np.int32)
    for b in range(8):
        zt[b, 0, cand[b]] = -30.0
    inp = {"target": zt, "draft": zd, "parents": np.full(kids, -1, np.int32), "cand": cand,
           "temperature": 1.0, "max_depth": 1}
    _check(inp, mode, seed=kids + 1, fill=rs.FILL_LEVEL)


def test_level_fill_without_room_on_the_draft_support():
    """Draft rows that exclude (-inf) half of the vocabulary, where the
    target keeps most of its mass: the level saturates the draft's support
    and the default fill places the rest, as in the oracle."""
    V, k, B = 512, 4, 64
    rng = np.random.default_rng(23)
    zt = rng.normal(0, 1, (B, k + 1, V)).astype(np.float32)
    zd = rng.normal(0, 1, (B, k + 1, V)).astype(np.float32)
    zt[:, :, V // 2:] += 8.0
    zd[:, :, V // 2:] = -np.inf
    cand = rng.integers(0, V // 2, (B, k)).astype(np.int32)
    for b in range(B):   # every candidate rejected: four shapings per sequence
        zt[b, 0, cand[b]] = -30.0
    # the first rejection at the root already finds no finite level
    no_room = 0
    for b in range(B):
        p0, q0 = sp_softmax(zt[b, 0].astype(np.float64)), sp_softmax(zd[b, 0].astype(np.float64))
        x0 = cand[b, 0]
        no_room += p0[q0 > 0].sum() - p0[x0] < q0[x0] - p0[x0]
    assert no_room > B // 2
    inp = {"target": zt, "draft": zd, "parents": np.full(k, -1, np.int32), "cand": cand,
           "temperature": 1.0, "max_depth": 1}
    g, o = _check(inp, rs.MODE_RESISPEC, seed=231, fill=rs.FILL_LEVEL)
    assert (o["rejects"] == k).all()
    o0 = P.run_oracle(zt, zd, inp["parents"], cand, 1.0, 231, 1, rs.MODE_RESISPEC)
    assert np.abs(o["dist"] - o0["dist"]).max() > 1e-5   # 30x the parity bound


def test_parity_level_fill_binary5_full_size():
    w = W.WORKLOADS["binary5-v151936-b64"]
    _sampled_parity(w, seed=35, call_seed=1006, rows=[1, 22, 40, 61], fill=rs.FILL_LEVEL)


def test_gpu_level_fill_million_draws_vs_enumerator():
    """The level fill on the GPU follows its own enumerated law (the
    enumerator finds the level by bisection)."""
    import torch
    V, k, n = 16, 3, 1_000_000
    rng = np.random.default_rng(7)
    zt = (2.0 * rng.standard_normal(V)).astype(np.float32)
    zd = (0.8 * zt + 1.2 * rng.standard_normal(V)).astype(np.float32)
    p, q = sp_softmax(zt.astype(np.float64)), sp_softmax(zd.astype(np.float64))
    cand = rng.choice(V, size=(n, k), p=q).astype(np.int32)
    toks, _ = rs.verify(P.to_device(np.broadcast_to(zt, (k + 1, V)).copy()),
                        P.to_device(np.broadcast_to(zd, (k + 1, V)).copy()),
                        torch.full((k,), -1, dtype=torch.int32, device="cuda"),
                        torch.as_tensor(cand, device="cuda"), 1.0, 99, max_depth=1,
                        seq_stride=0, fill=rs.FILL_LEVEL)
    counts = np.bincount(toks[:, 0].cpu().numpy(), minlength=V)
    dist, _ = en.single_position(p, q, k, en.MODE_RESISPEC, fill=1)
    dist0, _ = en.single_position(p, q, k, en.MODE_RESISPEC)
    assert chisq_pvalue(counts, dist)[0] > 1e-4
    assert np.abs(dist - dist0).max() > 1e-3 and chisq_pvalue(counts, dist0)[0] < 1e-8


@pytest.mark.parametrize("mode", MODES)
def test_diagnostics_match_oracle(mode):
    """Acceptance by candidate position (one position, 8 candidates) and the
    accepted length of a depth-4 chain with 4 candidates per position, from
    the kernel's outputs and from the oracle's on the same inputs, over the
    sequences without a near tie."""
    from paper_2608_24411_gb300 import diagnostics as dg
    for tree, B in ((("single", 8), 512), (("chain", 4, 4), 256)):
        w = W.Workload(name="diag", batch=B, vocab=32000, dtype="bf16", gen="zipf", scale=3.0,
                       slope=1.1, rho=0.8, temperature=1.0, tree=tree, steps=1)
        inp = W.make_inputs_np(w, seed=91, batch=B)
        g, o = _check(inp, mode, seed=92)
        clean = (o["accept_margin"] > P.ACCEPT_TIE) & (o["sample_margin"] > P.SAMPLE_TIE)
        if tree[0] == "single":
            pg = dg.accepted_position(g["accept_len"], g["nodes"], 8)[clean]
            po = dg.accepted_position(o["accept_len"], o["nodes"], 8)[clean]
            for a, b in zip(dg.position_rates(pg, 8), dg.position_rates(po, 8)):
                np.testing.assert_array_equal(a, b)
        else:
            assert (g["accept_len"][clean] + 1).mean() == (o["accept_len"][clean] + 1).mean()


def test_phase_counters():
    """Per-sequence cycle counters: filled for every sequence, no rejection
    phase when every first candidate is accepted (identical rows), a
    rejection phase when the target excludes every candidate."""
    import torch
    V, k, B = 4000, 4, 32
    rng = np.random.default_rng(3)
    z = rng.normal(0, 2, (B, k + 1, V)).astype(np.float32)
    cand = rng.integers(0, V, (B, k)).astype(np.int32)
    parents = np.full(k, -1, np.int32)
    for same in (True, False):
        zt = z.copy()
        if not same:
            for b in range(B):
                zt[b, 0, cand[b]] = -30.0
        cyc = torch.full((B, len(rs.PHASES)), -1, dtype=torch.int64, device="cuda")
        toks, alen = rs.verify(P.to_device(zt), P.to_device(z), torch.as_tensor(parents, device="cuda"),
                               torch.as_tensor(cand, device="cuda"), 1.0, 4, max_depth=1,
                               mode=rs.MODE_SPECINFER, out_phase=cyc)
        c = cyc.cpu().numpy()
        assert (c >= 0).all() and (c.sum(axis=1) > 0).all()
        rej = c[:, rs.PHASES.index("reject")]
        assert (rej == 0).all() if same else (rej > 0).all()
        assert (c[:, rs.PHASES.index("norm")] > 0).all() and (c[:, rs.PHASES.index("draw")] > 0).all()


def _check_drafting(inp, mode, seed, **kw):
    import torch
    zt, zd, pa, _ = _np_inputs_to_gpu(inp)
    D = int(inp["max_depth"])
    B, N = inp["cand"].shape
    drafted = torch.full((B, N), -7, dtype=torch.int32, device="cuda")
    g = P.run_gpu(zt, zd, pa, None, inp["temperature"], seed, D, mode=mode,
                  out_candidates=drafted, **kw)
    o = oracle.verify(inp["target"], inp["draft"], inp["parents"], inp["cand"],
                      inp["temperature"], seed, mode=mode, max_depth=D, want_dist=True,
                      draft_children=True)
    o["sample_margin"] = np.minimum(o["sample_margin"], o["draft_margin"])
    rep = P.compare(g, o)
    n, near = rep["sequences"], rep["mismatch_in_ties"]
    assert near <= max(2, 0.01 * n), (near, n)
    gd = drafted.cpu().numpy()
    clean = (o["accept_margin"] > P.ACCEPT_TIE) & (o["sample_margin"] > P.SAMPLE_TIE)
    np.testing.assert_array_equal(gd[clean], o["drafted"][clean])
    return gd, o


@pytest.mark.parametrize("mode", MODES)
@pytest.mark.parametrize("wl", ["tree60-v32000", "chain8x4-v128256-b16", "dyntree60-v32000"])
def test_parity_drafting(wl, mode):
    """Drafting mode: the kernel draws the children of every visited node
    from the node's draft distribution, then verifies them; tokens, accept
    lengths and drafted candidates against the oracle's drafting walk."""
    w = W.WORKLOADS[wl]
    inp = _inputs(w.name, 17, 256 if wl != "chain8x4-v128256-b16" else 16)
    gd, _ = _check_drafting(inp, mode, seed=170 + mode)
    assert (gd[:, :1] >= 0).all()   # the root's first child is always drawn


@pytest.mark.parametrize("mode", MODES)
@pytest.mark.parametrize("cluster,threads", [(1, 256), (1, 512), (2, 256), (2, 512)])
def test_parity_drafting_wide_fanout(cluster, threads, mode):
    """Drafting 16 children per node in one or two CTAs: a CTA draws more
    children than it has warps or single-row ring stages, so its draws run
    in batches (one warp per child); tokens, accept lengths and drafted
    candidates against the oracle's drafting walk."""
    w = dataclasses.replace(W.WORKLOADS["single-k16-v256000-b32"], vocab=20000,
                            name="single-k16-v20000")
    inp = W.make_inputs_np(w, seed=23, batch=64)
    gd, _ = _check_drafting(inp, mode, seed=230 + cluster, cluster_size=cluster,
                            block_threads=threads)
    assert (gd >= 0).all()   # a single position: every child is drawn


def test_gpu_drafted_candidates_follow_q():
    import torch
    V, k, n = 16, 3, 1_000_000
    rng = np.random.default_rng(8)
    zt = (2.0 * rng.standard_normal(V)).astype(np.float32)
    zd = (0.8 * zt + 1.2 * rng.standard_normal(V)).astype(np.float32)
    q = sp_softmax(zd.astype(np.float64))
    drafted = torch.full((n, k), -7, dtype=torch.int32, device="cuda")
    rs.verify(P.to_device(np.broadcast_to(zt, (k + 1, V)).copy()),
              P.to_device(np.broadcast_to(zd, (k + 1, V)).copy()),
              torch.full((k,), -1, dtype=torch.int32, device="cuda"), None, 1.0, 97,
              max_depth=1, seq_stride=0, out_candidates=drafted)
    d = drafted.cpu().numpy()
    assert (d[:, 0] >= 0).all()
    assert chisq_pvalue(np.bincount(d[:, 0], minlength=V), q)[0] > 1e-4


def test_specinfer_residual_ill_conditioned():
    """SpecInfer rows whose residual mass N = prod S_j is small: a draft
    close to the target (rho 0.98) and 6 forced rejections of tokens the
    target excludes (draft ranks 300-305) drive 1 / N into the thousands on
    some rows, where the residual (p - C q)_+ / N magnifies any relative
    error of its sums and exponentials by p / N; the kernel's double-float
    evaluation meets the flat 1e-6 on every row."""
    V, kids, B = 32000, 6, 64
    rng = np.random.default_rng(77)
    zt = (3.0 * rng.normal(0, 1, (B, kids + 1, V))
          - np.log(rng.permuted(np.tile(np.arange(1, V + 1), (B, kids + 1, 1)), axis=2)))
    zd = 0.98 * zt + np.sqrt(1 - 0.98 ** 2) * 3.0 * rng.normal(0, 1, zt.shape)
    zt, zd = zt.astype(np.float32), zd.astype(np.float32)
    cand = np.argsort(-zd[:, 0], axis=1)[:, 300:300 + kids].astype(np.int32)
    for b in range(B):
        zt[b, 0, cand[b]] = -30.0          # the target all but excludes them: every test rejects
    inp = {"target": zt, "draft": zd, "parents": np.full(kids, -1, np.int32), "cand": cand,
           "temperature": 1.0, "max_depth": 1}
    g, o = _check(inp, rs.MODE_SPECINFER, seed=5, kernel="stream")
    assert (o["rejects"] == kids).all()
    assert o["cond"].max() > 1000.0, o["cond"].max()   # 1 / N: the conditioning under test
