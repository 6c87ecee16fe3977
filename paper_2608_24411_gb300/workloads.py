"""Seeded synthetic inputs for the verification walk.

This module draws inputs only: draft trees, target/draft logits and the
candidate tokens the drafter would have proposed.  It holds none of the
verification arithmetic (no normaliser, no accept test, no shaping, no
sampler); candidates are drawn from the tempered draft softmax with the
Gumbel-max identity, argmax_x (z_d(x)/T + G_x) with G_x i.i.d. Gumbel(0, 1),
so no softmax is ever formed here.

Logit recipes (stand-ins for the target / draft models the paper runs on
its datasets, Sec. 6.1):

* ``gauss``: z_t = s * N(0,1), z_d = rho * z_t + sqrt(1 - rho^2) * s * N(0,1).
* ``zipf``:  z_t = s * N(0,1) - a * log(rank), rank a fresh random
  permutation of 1..V per row (Zipf-like head, Gaussian noise),
  z_d = rho * z_t + sqrt(1 - rho^2) * s * N(0,1).

Tree shapes (the paper's dXbY trees and batch-sampling chains, Sec. 3):
``levels`` (every node of level l has b[l] children, BFS numbering),
``chain`` (k siblings per level, level l+1 hangs below sibling 0 of level l)
and ``single`` (k siblings of the root), one tree for every sequence; and
``random`` (a tree of N nodes per sequence, as dynamic-tree drafters build
them: node c hangs below a node drawn among the root and the earlier nodes
less than Dmax deep, with weight 2^-depth, so the top levels are bushy and
the deep ones thin; nodes are numbered in creation order).
"""
from __future__ import annotations

import math
from dataclasses import dataclass, field

import numpy as np

# ------------------------------------------------------------------ trees


def tree_levels(branching) -> np.ndarray:
    parents = []
    frontier = [-1]
    for b in branching:
        nxt = []
        for p in frontier:
            for _ in range(int(b)):
                parents.append(p)
                nxt.append(len(parents) - 1)
        frontier = nxt
    return np.asarray(parents, dtype=np.int32)


def tree_chain(depth: int, k: int) -> np.ndarray:
    parents = []
    spine = -1
    for _ in range(int(depth)):
        first = len(parents)
        parents.extend([spine] * int(k))
        spine = first
    return np.asarray(parents, dtype=np.int32)


def tree_single(k: int) -> np.ndarray:
    return np.full(int(k), -1, dtype=np.int32)


def tree_depth(parents) -> int:
    parents = np.asarray(parents)
    depth = np.zeros(parents.size, dtype=np.int64)
    for c, p in enumerate(parents):
        depth[c] = 1 if p < 0 else depth[p] + 1
    return int(depth.max()) if parents.size else 0


def tree_random(rng: np.random.Generator, B: int, N: int, dmax: int) -> np.ndarray:
    """[B, N] int32 parents: one random tree of N nodes (depth <= dmax) per
    sequence."""
    out = np.zeros((int(B), int(N)), dtype=np.int32)
    for b in range(int(B)):
        depth = [0]          # the root, then node c at index c + 1
        for c in range(int(N)):
            cand = [i for i, d in enumerate(depth) if d < dmax]
            w = np.asarray([0.5 ** depth[i] for i in cand])
            pick = cand[int(rng.choice(len(cand), p=w / w.sum()))]
            out[b, c] = pick - 1
            depth.append(depth[pick] + 1)
    return out


def per_sequence_tree(spec) -> bool:
    return spec[0] == "random"


def make_tree(spec) -> np.ndarray:
    kind = spec[0]
    if kind == "levels":
        return tree_levels(spec[1])
    if kind == "chain":
        return tree_chain(spec[1], spec[2])
    if kind == "single":
        return tree_single(spec[1])
    raise ValueError(f"unknown tree kind {kind!r}")


# ------------------------------------------------------------------ workloads


@dataclass(frozen=True)
class Workload:
    name: str
    batch: int
    vocab: int
    dtype: str            # "f32" or "bf16"
    gen: str              # "gauss" or "zipf"
    scale: float
    slope: float
    rho: float
    temperature: float
    tree: tuple
    steps: int
    note: str = ""
    extra: dict = field(default_factory=dict)

    @property
    def per_sequence_tree(self) -> bool:
        return per_sequence_tree(self.tree)

    @property
    def parents(self) -> np.ndarray:
        """The shared tree ([N]); per-sequence trees come with the inputs."""
        if self.per_sequence_tree:
            raise ValueError(f"{self.name}: a tree per sequence, drawn with the inputs")
        return make_tree(self.tree)

    @property
    def num_nodes(self) -> int:
        return int(self.tree[1]) if self.per_sequence_tree else int(self.parents.size)

    @property
    def max_depth(self) -> int:
        return int(self.tree[2]) if self.per_sequence_tree else tree_depth(self.parents)

    @property
    def elem_bytes(self) -> int:
        return 4 if self.dtype == "f32" else 2


def _w(**kw) -> Workload:
    return Workload(**kw)


WORKLOADS = {
    "tiny-chain-v64": _w(
        name="tiny-chain-v64", batch=1, vocab=64, dtype="f32", gen="gauss", scale=2.0,
        slope=0.0, rho=0.8, temperature=1.0, tree=("chain", 4, 3), steps=10_000,
        note="chain depth 4, k=3; z_t~N(0,4), z_d=0.8 z_t+0.6*2 N(0,1)"),
    "tree60-v32000": _w(
        name="tree60-v32000", batch=1, vocab=32000, dtype="bf16", gen="zipf", scale=3.0,
        slope=1.1, rho=0.9, temperature=1.0, tree=("levels", (4, 2, 2, 1, 1)), steps=1000),
    "chain8x4-v128256-b16": _w(
        name="chain8x4-v128256-b16", batch=16, vocab=128256, dtype="bf16", gen="zipf",
        scale=3.0, slope=1.1, rho=0.8, temperature=0.7, tree=("chain", 4, 8), steps=1000),
    "binary5-v151936-b64": _w(
        name="binary5-v151936-b64", batch=64, vocab=151936, dtype="f32", gen="zipf",
        scale=4.0, slope=1.0, rho=0.8, temperature=1.0, tree=("levels", (2, 2, 2, 2, 2)),
        steps=500, note="rho swept over {0.5, 0.8, 0.95}; 0.8 is the default"),
}
WORKLOADS["dyntree60-v32000"] = _w(
    name="dyntree60-v32000", batch=64, vocab=32000, dtype="bf16", gen="zipf", scale=3.0,
    slope=1.1, rho=0.9, temperature=1.0, tree=("random", 60, 6), steps=200,
    note="a random 60-node tree of depth <= 6 per sequence (dynamic trees)")
WORKLOADS["dyntree60-v128256-b64"] = _w(
    name="dyntree60-v128256-b64", batch=64, vocab=128256, dtype="bf16", gen="zipf",
    scale=3.0, slope=1.1, rho=0.8, temperature=1.0, tree=("random", 60, 6), steps=200,
    note="a random 60-node tree of depth <= 6 per sequence (dynamic trees)")
for _b in (32, 128):
    for _k in (2, 4, 8, 16):
        WORKLOADS[f"single-k{_k}-v256000-b{_b}"] = _w(
            name=f"single-k{_k}-v256000-b{_b}", batch=_b, vocab=256000, dtype="bf16",
            gen="zipf", scale=3.0, slope=1.1, rho=0.85, temperature=1.0,
            tree=("single", _k), steps=200)
    WORKLOADS[f"tree488-v256000-b{_b}"] = _w(
        name=f"tree488-v256000-b{_b}", batch=_b, vocab=256000, dtype="bf16", gen="zipf",
        scale=3.0, slope=1.1, rho=0.85, temperature=1.0,
        tree=("levels", (8, 4, 2, 2, 1, 1)), steps=200)


def with_rho(w: Workload, rho: float) -> Workload:
    d = dict(w.__dict__)
    d["rho"] = float(rho)
    d["name"] = f"{w.name}-rho{rho:g}"
    return Workload(**d)


# ------------------------------------------------------------------ numpy (host)


def f32_to_bf16_bits(x: np.ndarray) -> np.ndarray:
    """Round float32 to bfloat16 (round to nearest even), as uint16 bits."""
    x = np.ascontiguousarray(x, dtype=np.float32)
    u = x.view(np.uint32).astype(np.uint64)
    bias = ((u >> 16) & 1) + 0x7FFF
    out = ((u + bias) >> 16).astype(np.uint16)
    nan = np.isnan(x)
    out[nan] = 0x7FC0
    return out


def bf16_bits_to_f32(b: np.ndarray) -> np.ndarray:
    return (np.asarray(b, dtype=np.uint16).astype(np.uint32) << 16).view(np.float32)


def logits_np(rng: np.random.Generator, rows: int, V: int, gen: str, scale: float,
              slope: float, rho: float):
    """(z_t, z_d) float32 arrays of shape [rows, V]."""
    zt = scale * rng.standard_normal((rows, V))
    if gen == "zipf":
        rank = rng.permuted(np.broadcast_to(np.arange(1, V + 1, dtype=np.float64), (rows, V)),
                            axis=1)
        zt = zt - slope * np.log(rank)
    elif gen != "gauss":
        raise ValueError(gen)
    zd = rho * zt + math.sqrt(max(0.0, 1.0 - rho * rho)) * scale * rng.standard_normal((rows, V))
    return zt.astype(np.float32), zd.astype(np.float32)


def gumbel_argmax_np(rng: np.random.Generator, z_rows: np.ndarray, T: float) -> np.ndarray:
    """One draw per row from softmax(z/T) via argmax(z/T + Gumbel)."""
    u = rng.random(z_rows.shape)
    g = -np.log(-np.log(np.maximum(u, 1e-300)))
    return np.argmax(z_rows.astype(np.float64) / T + g, axis=-1).astype(np.int32)


def candidates_np(rng, draft_f32: np.ndarray, parents: np.ndarray, T: float) -> np.ndarray:
    """cand[b, c] drawn from the tempered draft row of c's parent.

    ``draft_f32``: [B, N+1, V] float32 (row 0 = root, row j+1 = node j);
    ``parents``: [N] (shared tree) or [B, N] (a tree per sequence).
    """
    B = draft_f32.shape[0]
    N = parents.shape[-1]
    if N == 0:
        return np.zeros((B, 0), dtype=np.int32)
    parent_rows = parents.astype(np.int64) + 1
    if parents.ndim == 2:
        z = np.take_along_axis(draft_f32, parent_rows[:, :, None], axis=1)  # [B, N, V]
    else:
        z = draft_f32[:, parent_rows, :]                 # [B, N, V]
    return gumbel_argmax_np(rng, z, T).reshape(B, N)


def make_inputs_np(w: Workload, seed: int, batch: int | None = None, rho: float | None = None):
    """Host inputs for a workload: dict with target/draft ([B, N+1, V] float32
    or uint16 bf16 bits), parents, cand, temperature, max_depth."""
    rng = np.random.default_rng(seed)
    B = w.batch if batch is None else int(batch)
    if w.per_sequence_tree:
        parents = tree_random(rng, B, w.tree[1], w.tree[2])
    else:
        parents = w.parents
    N = parents.shape[-1]
    zt, zd = logits_np(rng, B * (N + 1), w.vocab, w.gen, w.scale, w.slope,
                       w.rho if rho is None else rho)
    zt = zt.reshape(B, N + 1, w.vocab)
    zd = zd.reshape(B, N + 1, w.vocab)
    if w.dtype == "bf16":
        zt_s, zd_s = f32_to_bf16_bits(zt), f32_to_bf16_bits(zd)
        zd_for_draw = bf16_bits_to_f32(zd_s)
    else:
        zt_s, zd_s = zt, zd
        zd_for_draw = zd
    cand = candidates_np(rng, zd_for_draw, parents, w.temperature)
    return dict(target=zt_s, draft=zd_s, parents=parents, cand=cand,
                temperature=w.temperature, max_depth=w.max_depth, dtype=w.dtype)


def path_rows_np(seed: int, V: int, scale: float, rho: float):
    """rows(path) -> (z_t, z_d) float32 rows that depend only on the token
    path from the root, for joint (multi-level) exactness checks."""
    cache = {}

    def rows(path):
        key = tuple(int(t) for t in path)
        if key not in cache:
            rng = np.random.default_rng([int(seed), len(key)] + [t + 1 for t in key])
            zt = scale * rng.standard_normal(V)
            zd = rho * zt + math.sqrt(1.0 - rho * rho) * scale * rng.standard_normal(V)
            cache[key] = (zt.astype(np.float32), zd.astype(np.float32))
        return cache[key]

    return rows


def make_path_inputs_np(seed: int, parents: np.ndarray, B: int, V: int, T: float,
                        scale: float = 1.0, rho: float = 0.5):
    """B independent draws of one tree whose rows are a function of the token
    path (duplicate siblings share rows).  Returns (target, draft, cand,
    rows_fn) with target/draft float32 [B, N+1, V]."""
    rng = np.random.default_rng(seed)
    rows = path_rows_np(seed + 7919, V, scale, rho)
    N = parents.size
    target = np.zeros((B, N + 1, V), np.float32)
    draft = np.zeros((B, N + 1, V), np.float32)
    cand = np.zeros((B, N), np.int32)
    root_t, root_d = rows(())
    target[:, 0] = root_t
    draft[:, 0] = root_d
    gumbel = -np.log(-np.log(np.maximum(rng.random((B, N, V)), 1e-300)))
    for b in range(B):
        node_path = {}
        for c in range(N):
            pa = int(parents[c])
            pp = () if pa < 0 else node_path[pa]
            _, pd = rows(pp)
            x = int(np.argmax(pd.astype(np.float64) / T + gumbel[b, c]))
            cand[b, c] = x
            node_path[c] = pp + (x,)
            zt, zd = rows(node_path[c])
            target[b, c + 1] = zt
            draft[b, c + 1] = zd
    return target, draft, cand, rows


# ------------------------------------------------------------------ torch (device)


def make_inputs_torch(w: Workload, seed: int, device, batch: int | None = None,
                      rho: float | None = None, row_chunk: int = 256):
    """Device inputs for the large workloads, drawn with a seeded torch
    generator on ``device``; same recipe as :func:`make_inputs_np`."""
    import torch

    g = torch.Generator(device=device)
    g.manual_seed(int(seed))
    B = w.batch if batch is None else int(batch)
    if w.per_sequence_tree:
        parents = tree_random(np.random.default_rng([int(seed), 1]), B, w.tree[1], w.tree[2])
    else:
        parents = w.parents
    N = parents.shape[-1]
    V = w.vocab
    rho = w.rho if rho is None else float(rho)
    tdtype = torch.float32 if w.dtype == "f32" else torch.bfloat16
    rows = B * (N + 1)
    target = torch.empty((rows, V), dtype=tdtype, device=device)
    draft = torch.empty((rows, V), dtype=tdtype, device=device)
    noise_w = math.sqrt(max(0.0, 1.0 - rho * rho)) * w.scale
    for r0 in range(0, rows, row_chunk):
        r1 = min(rows, r0 + row_chunk)
        n = r1 - r0
        zt = w.scale * torch.randn((n, V), generator=g, device=device)
        if w.gen == "zipf":
            rank = torch.argsort(torch.rand((n, V), generator=g, device=device), dim=1) + 1
            zt = zt - w.slope * torch.log(rank.to(torch.float32))
            del rank
        zd = rho * zt + noise_w * torch.randn((n, V), generator=g, device=device)
        target[r0:r1] = zt.to(tdtype)
        draft[r0:r1] = zd.to(tdtype)
        del zt, zd
    target = target.view(B, N + 1, V)
    draft = draft.view(B, N + 1, V)
    cand = torch.zeros((B, max(N, 0)), dtype=torch.int32, device=device)
    if N:
        prow = torch.as_tensor(parents.astype(np.int64) + 1, device=device)
        node_chunk = max(1, (1 << 28) // max(1, B * V))
        bidx = torch.arange(B, device=device)[:, None]
        for c0 in range(0, N, node_chunk):
            c1 = min(N, c0 + node_chunk)
            if prow.dim() == 2:
                z = draft[bidx, prow[:, c0:c1], :].to(torch.float32) / w.temperature
            else:
                z = draft[:, prow[c0:c1], :].to(torch.float32) / w.temperature
            u = torch.rand(z.shape, generator=g, device=device).clamp_min_(1e-30)
            z.add_(-torch.log(-torch.log(u)))
            cand[:, c0:c1] = torch.argmax(z, dim=-1).to(torch.int32)
            del z, u
    return dict(target=target, draft=draft,
                parents=torch.as_tensor(np.ascontiguousarray(parents), device=device),
                parents_np=parents, cand=cand, temperature=w.temperature,
                max_depth=w.max_depth, dtype=w.dtype)
