#!/usr/bin/env python3
"""Benchmark of the fused ResiSpec verification kernel on GB300.

One step = one resispec_verify call over one batch of synthetic input (the
whole hot path: tempered normaliser, accept tests, residual shaping, tree
walk, residual/bonus sampling, Philox).  Default workload: B = 64 sequences,
V = 151936, fp32 logits, full binary tree of depth 5 (62 nodes per
sequence), Zipf-plus-Gaussian logits (slope 1.0, scale 4, rho 0.8), T = 1.0,
ResiSpec mode.

Prints one JSON line (rank 0).  `value` is verified tree nodes per second
over all ranks (B * N per call); the roofline object reports algorithmic
logit bytes (only the rows the walk visits) per launch over the measured
launch time against the measured HBM copy bandwidth.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]
"""
from __future__ import annotations

import argparse
import hashlib
import json
import math
import os
import re
import statistics
import subprocess
import sys
import tempfile
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

METRIC = ("verified tree nodes/sec and HBM GB/s (fraction of 8 TB/s) at 1 GB300 vs CPU oracle")
NOMINAL_HBM_GBS = 8000.0
FALLBACK_HBM_GBS = 6800.0
L2_BYTES = 129 * 1024 * 1024


def parse_args(argv=None):
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=2000)
    ap.add_argument("--warmup", type=int, default=20)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--workload", default="binary5-v151936-b64")
    ap.add_argument("--rho", type=float, default=None)
    ap.add_argument("--batch", type=int, default=None, help="override the workload's batch")
    ap.add_argument("--mode", choices=["resispec", "specinfer"], default="resispec")
    ap.add_argument("--z-rule", choices=["alg1", "applied"], default="alg1",
                    help="ResiSpec budget: Algorithm 1's gap, or the Z_applied heuristic")
    ap.add_argument("--proxy-denominator", action="store_true",
                    help="ResiSpec variant: each rejection's proxy becomes the test denominator")
    ap.add_argument("--fill", choices=["capacity", "level"], default="capacity",
                    help="ResiSpec variant of GetProxy's deficit fill: in proportion to the "
                         "capacity (default) or the draft raised to a level")
    ap.add_argument("--draft", action="store_true",
                    help="drafting mode: the kernel draws the visited nodes' children from q")
    ap.add_argument("--pool", type=int, default=0, help="input sets rotated between steps (0 = auto)")
    ap.add_argument("--cluster-size", type=int, default=0)
    ap.add_argument("--block-threads", type=int, default=0)
    ap.add_argument("--kernel", choices=["auto", "resident", "stream"], default="auto")
    ap.add_argument("--e2e-steps", type=int, default=12)
    ap.add_argument("--cpu-seqs", type=int, default=16)
    ap.add_argument("--cpu-seconds", type=float, default=12.0)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-clocks", action="store_true")
    ap.add_argument("--seed", type=int, default=1234)
    return ap.parse_args(argv)


def measured_peak():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            d = json.load(f)
        return float(d["hbm_gbs"]), "measured"
    except Exception:
        return FALLBACK_HBM_GBS, "fallback"


def kernel_source_digest(csrc=None):
    """Digest of the kernel sources (`csrc/`) with their comments removed:
    the committed ncu counters are keyed to the code they measured, and a
    change of comments alone does not invalidate them."""
    h = hashlib.sha256()
    csrc = csrc or os.path.join(ROOT, "paper_2608_24411_gb300", "csrc")
    for name in sorted(os.listdir(csrc)):
        with open(os.path.join(csrc, name), encoding="utf-8") as f:
            code = f.read()
        code = re.sub(r"/\*.*?\*/", " ", code, flags=re.S)
        code = re.sub(r"//[^\n]*", "", code)
        code = "\n".join(line.rstrip() for line in code.splitlines() if line.strip())
        h.update(name.encode())
        h.update(code.encode())
    return h.hexdigest()[:16]


def profiled_traffic(kernel, workload, alg_bytes_per_launch):
    """DRAM bytes per launch: the committed ncu summary of this kernel on
    this workload gives DRAM bytes per algorithmic byte (measured on a
    smaller case of the same kernel); traffic grows with the rows visited,
    so it is scaled by this run's algorithmic bytes per launch.  None unless
    the summary was taken on the current kernel source."""
    path = os.path.join(ROOT, "profiles", f"{kernel}_kernel_{workload}.md")
    if not os.path.exists(path):
        return None
    text = open(path).read()
    m_src = re.search(r"kernel_source_digest:\s*([0-9a-f]+)", text)
    m_tr = re.search(r"dram_bytes_per_alg_byte:\s*([0-9.eE+]+)", text)
    if not m_src or not m_tr or m_src.group(1) != kernel_source_digest():
        return None
    return float(m_tr.group(1)) * alg_bytes_per_launch


# ------------------------------------------------------------------ clocks


class ClockSampler:
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, device_index, enabled=True):
        self.proc = None
        self.path = None
        self.dev = device_index
        if not enabled:
            return
        try:
            fd, self.path = tempfile.mkstemp(prefix=f"resispec_clocks_rank{device_index}_",
                                             suffix=".csv")
            self.fh = os.fdopen(fd, "w")
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--id={device_index}", f"--query-gpu={self.FIELDS}",
                 "--format=csv,noheader,nounits", "-lms", "100"],
                stdout=self.fh, stderr=subprocess.DEVNULL)
        except Exception:
            self.proc = None
            if self.path:
                try:
                    self.fh.close()
                    os.unlink(self.path)
                except (OSError, AttributeError):
                    pass

    def stop(self):
        if self.proc is None:
            return None
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except Exception:
            self.proc.kill()
        self.fh.close()
        sm, mx, reasons = [], None, set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for line in open(self.path):
            parts = [p.strip() for p in line.split(",")]
            if len(parts) < 9:
                continue
            try:
                sm.append(float(parts[1]))
                mx = float(parts[2])
            except ValueError:
                continue
            for n, v in zip(names, parts[5:9]):
                if v.lower().startswith("active"):
                    reasons.add(n)
        try:
            os.unlink(self.path)
        except OSError:
            pass
        if not sm:
            return None
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": mx, "reasons": sorted(reasons),
                "samples": len(sm)}


# ------------------------------------------------------------------ helpers


def has_children(parents_np):
    """[N + 1] (one tree) or [B, N + 1] (a tree per sequence): whether the
    root (index 0) / node j (index j + 1) has children."""
    p = np.asarray(parents_np)
    if p.ndim == 1:
        h = np.zeros(p.size + 1, dtype=bool)
        h[p[p >= -1] + 1] = True
        return h
    h = np.zeros((p.shape[0], p.shape[1] + 1), dtype=bool)
    for b in range(p.shape[0]):
        h[b, p[b] + 1] = True
    return h


def rows_visited(nodes, accept_len, haschild):
    """Logit rows each sequence read: 2 per visited node with children
    (target + draft), 1 for a visited node without children (bonus: target
    only).  Visited nodes are the root and every accepted node."""
    a = accept_len.astype(np.int64)
    D = nodes.shape[1]
    hc = haschild if haschild.ndim == 2 else np.broadcast_to(haschild, (a.size, haschild.size))
    rows = np.where(hc[:, 0], 2, 1).astype(np.int64)
    for d in range(D):
        mask = a > d
        if not mask.any():
            break
        nd = nodes[mask, d]
        rows[mask] += np.where(hc[mask, nd + 1], 2, 1)
    return rows


def oracle_variant(args) -> dict:
    """The oracle's switches for the verification rule the run measures."""
    return dict(z_rule=1 if args.z_rule == "applied" else 0, denom_update=args.proxy_denominator,
                fill=1 if args.fill == "level" else 0, draft_children=args.draft)


def cpu_oracle_rate(w, target_h, draft_h, parents, cand_h, seq_ids, mode, seconds, seed0,
                    variant=None):
    """Time the fp64 oracle as it stands on this host's cores over a bounded
    sample; returns (nodes/s, threads, sample description)."""
    import oracle
    variant = variant or {}
    S = cand_h.shape[0]
    threads = min(os.cpu_count() or 1, S)
    # one thread on the first (at most two) sequences: the per-core rate
    s1 = min(2, S)
    p1 = parents[:s1] if np.asarray(parents).ndim == 2 else parents
    t1 = time.perf_counter()
    oracle.verify(target_h[:s1], draft_h[:s1], p1, cand_h[:s1], w.temperature, seed0,
                  mode=mode, max_depth=w.max_depth, seq_ids=seq_ids[:s1], nthreads=1, **variant)
    one_thread = s1 * w.num_nodes / (time.perf_counter() - t1)
    reps, t0 = 0, time.perf_counter()
    while True:
        oracle.verify(target_h, draft_h, parents, cand_h, w.temperature, seed0 + reps, mode=mode,
                      max_depth=w.max_depth, seq_ids=seq_ids, nthreads=threads, **variant)
        reps += 1
        el = time.perf_counter() - t0
        if el >= seconds or reps >= 200:
            break
    nodes = reps * S * w.num_nodes
    sample = (f"{reps} calls x {S} sequences of {w.name} (rows copied to host), "
              f"{nodes} verified nodes in {el:.2f} s")
    return nodes / el, threads, sample, one_thread


TIE_LEVELS = (1e-5, 1e-6, 1e-7)


def parity_sample(g, o):
    """GPU outputs g against the oracle's o on the same sequences: the
    near-tie counts (oracle margins, fp64 accept decisions) at 1e-5 / 1e-6 /
    1e-7 and the sequences whose accepted tokens, accept length, accepted
    node ids, rejection count or final token differ, inside and outside the
    tie band (accept margin <= 1e-5 or final-draw margin <= 1e-6)."""
    near = (o["accept_margin"] <= TIE_LEVELS[0]) | (o["sample_margin"] <= TIE_LEVELS[1])
    D = o["nodes"].shape[1]
    same = (g["accept_len"] == o["accept_len"]) & (g["tokens"] == o["tokens"]).all(axis=1)
    same &= (g["rejects"] == o["rejects"])
    if D:
        same &= (g["nodes"][:, :D] == o["nodes"]).all(axis=1)
    counts = {}
    for t in TIE_LEVELS:
        counts[f"accept<={t:g}"] = int((o["accept_margin"] <= t).sum())
        counts[f"sample<={t:g}"] = int((o["sample_margin"] <= t).sum())
    return {"sequences": int(len(same)), "near_tie": counts,
            "mismatch_in_ties": int((~same & near).sum()),
            "mismatch_outside_ties": int((~same & ~near).sum())}


def cpu_model() -> str:
    """The host CPU's model name (lscpu's, or /proc/cpuinfo's), else the
    machine type."""
    try:
        out = subprocess.run(["lscpu"], capture_output=True, text=True, timeout=10).stdout
        for line in out.splitlines():
            if line.startswith("Model name:"):
                return line.split(":", 1)[1].strip()
    except (OSError, subprocess.SubprocessError):
        pass
    try:
        for line in open("/proc/cpuinfo"):
            if line.startswith("model name"):
                return line.split(":", 1)[1].strip()
    except OSError:
        pass
    import platform
    return platform.machine()


# ------------------------------------------------------------------ ranks


def rank_layout():
    """(rank, local rank, world size) from the launcher's environment."""
    return (int(os.environ.get("RANK", "0")), int(os.environ.get("LOCAL_RANK", "0")),
            int(os.environ.get("WORLD_SIZE", "1")))


def replica_seed(seed, rank, i):
    """Seed of input set i on `rank`: every replica verifies its own data
    (weak scaling, no exchange between ranks)."""
    return seed + 7919 * rank + 31 * i


class RankGroup:
    """Barrier and scalar reductions over the ranks of a replicas run (one
    process per GPU).  The path has no data exchange between ranks: these
    calls only bracket the timed region and combine its timings.  With
    dist None (one process) every call is local."""

    def __init__(self, dist=None, device=None):
        self.dist = dist
        self.device = device

    def barrier(self):
        if self.dist is not None:
            self.dist.barrier()

    def _reduce(self, x, op):
        if self.dist is None:
            return float(x)
        import torch
        t = torch.tensor([float(x)], dtype=torch.float64, device=self.device)
        self.dist.all_reduce(t, op=op)
        return float(t.item())

    def max(self, x):
        return self._reduce(x, None if self.dist is None else self.dist.ReduceOp.MAX)

    def sum(self, x):
        return self._reduce(x, None if self.dist is None else self.dist.ReduceOp.SUM)


def whole_job_rate(group, units_this_rank, elapsed_ms_this_rank):
    """Whole-job throughput: the units all ranks processed over the slowest
    rank's time (max over ranks, the timed region of every rank bracketed by
    a barrier)."""
    total = group.sum(units_this_rank)
    slowest_ms = group.max(elapsed_ms_this_rank)
    return total / (slowest_ms / 1e3), slowest_ms


# ------------------------------------------------------------------ reference arm


def run_reference(args):
    """The oracle as it stands on the host cores, on this arm's workload."""
    import oracle
    from paper_2608_24411_gb300 import workloads as W
    rank, _, _ = rank_layout()
    if rank != 0:
        return 0  # under torchrun rank 0 alone times the oracle
    w = W.WORKLOADS[args.workload]
    if args.rho is not None:
        w = W.with_rho(w, args.rho)
    mode = oracle.MODE_SPECINFER if args.mode == "specinfer" else oracle.MODE_RESISPEC
    S = max(1, args.cpu_seqs)
    inp = W.make_inputs_np(w, seed=args.seed, batch=S)
    seq_ids = np.arange(S, dtype=np.int32)
    threads = min(os.cpu_count() or 1, S)

    def step(i):
        oracle.verify(inp["target"], inp["draft"], inp["parents"], inp["cand"], w.temperature,
                      args.seed + i, mode=mode, max_depth=w.max_depth, seq_ids=seq_ids,
                      nthreads=threads, **oracle_variant(args))

    for i in range(max(0, args.warmup)):
        step(i)
    t0 = time.perf_counter()
    for i in range(args.steps):
        step(args.warmup + i)
    el = time.perf_counter() - t0
    value = args.steps * S * w.num_nodes / el
    line = {
        "impl": "reference", "metric": METRIC, "value": value, "unit": "nodes/s",
        "n_gpus": args.gpus, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": 1e3 * el / max(1, args.steps), "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "config": {"workload": w.name, "batch_per_step": S, "vocab": w.vocab,
                   "nodes_per_seq": w.num_nodes, "mode": args.mode, "rho": w.rho,
                   "z_rule": args.z_rule, "proxy_denominator": args.proxy_denominator,
                   "fill": args.fill, "draft": args.draft},
        "cpu_baseline": {"value": value, "unit": "nodes/s", "cores": threads, "kind": "oracle",
                         "sample": f"{S} sequences of {w.name} per step (host inputs)",
                         "cpu_model": cpu_model(), "nproc": os.cpu_count()},
        "e2e": {"value": value, "unit": "nodes/s", "h2d_bytes_per_step": 0,
                "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)
    return 0


# ------------------------------------------------------------------ our arm


def run_ours(args):
    import torch
    import paper_2608_24411_gb300 as rs
    from paper_2608_24411_gb300 import workloads as W

    rank, local, world = rank_layout()
    if world != args.gpus and world > 1:
        raise SystemExit(f"--gpus {args.gpus} but WORLD_SIZE {world}")
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    dist = None
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", device_id=dev)
    group = RankGroup(dist, dev)
    barrier, max_over_ranks, sum_over_ranks = group.barrier, group.max, group.sum

    rs.build()
    rs.load_library()
    w = W.WORKLOADS[args.workload]
    if args.rho is not None:
        w = W.with_rho(w, args.rho)
    mode = rs.MODE_SPECINFER if args.mode == "specinfer" else rs.MODE_RESISPEC
    B, N, V, D = (args.batch or w.batch), w.num_nodes, w.vocab, w.max_depth
    es = w.elem_bytes
    set_bytes = 2 * B * (N + 1) * V * es
    pool = args.pool or max(2, min(8, math.ceil(4 * L2_BYTES / max(1, 2 * B * V * es))))
    sets = [W.make_inputs_torch(w, seed=replica_seed(args.seed, rank, i), device=dev, batch=B)
            for i in range(pool)]
    haschild = [has_children(s["parents_np"]) for s in sets]
    K, Wm = args.steps, args.warmup
    outs = [(torch.empty((B, D + 1), dtype=torch.int32, device=dev),
             torch.empty((B,), dtype=torch.int32, device=dev),
             torch.empty((B, max(D, 1)), dtype=torch.int32, device=dev)) for _ in range(K)]
    status = torch.zeros((1,), dtype=torch.int32, device=dev)
    kernel = None if args.kernel == "auto" else args.kernel
    z_rule = rs.Z_RULE_APPLIED if args.z_rule == "applied" else rs.Z_RULE_ALG1
    fill = rs.FILL_LEVEL if args.fill == "level" else rs.FILL_CAPACITY
    kw = dict(max_depth=D, mode=mode, cluster_size=args.cluster_size,
              block_threads=args.block_threads, status=status, kernel=kernel, z_rule=z_rule,
              proxy_denominator=args.proxy_denominator, fill=fill)
    stream = torch.cuda.current_stream(dev)
    plan = rs.plan(B, N, V, D, w.dtype, cluster_size=args.cluster_size,
                   block_threads=args.block_threads,
                   kernel="stream" if (args.draft and kernel is None) else kernel,
                   z_rule=z_rule, proxy_denominator=args.proxy_denominator, fill=fill)

    drafted = torch.empty((B, N), dtype=torch.int32, device=dev) if args.draft else None

    def launch(i, out):
        s = sets[i % pool]
        rs.verify(s["target"], s["draft"], s["parents"], None if args.draft else s["cand"],
                  w.temperature, args.seed + i, out_tokens=out[0], out_accept_len=out[1],
                  out_nodes=out[2], stream=stream, out_candidates=drafted, **kw)

    for i in range(Wm):
        launch(i, outs[i % K])
    torch.cuda.synchronize()

    ev = [torch.cuda.Event(enable_timing=True) for _ in range(K + 1)]
    clocks = ClockSampler(local, enabled=not args.no_clocks)
    time.sleep(0.3 if not args.no_clocks else 0)
    barrier()
    torch.cuda.synchronize()
    wall0 = time.perf_counter()
    ev[0].record(stream)
    for i in range(K):
        launch(Wm + i, outs[i])
        ev[i + 1].record(stream)
    torch.cuda.synchronize()
    barrier()
    wall = time.perf_counter() - wall0
    clk = clocks.stop()
    launch_ms = [ev[i].elapsed_time(ev[i + 1]) for i in range(K)]
    value, elapsed_ms = whole_job_rate(group, float(K * B * N), ev[0].elapsed_time(ev[K]))
    if int(status.item()) & ~rs.INFO_DEGENERATE:
        raise SystemExit(f"kernel reported data errors: status {int(status.item())}")

    alg_bytes = 0
    emitted = 0
    accepted = 0
    rows_read = 0
    for i in range(K):
        alen = outs[i][1].cpu().numpy()
        nodes = outs[i][2].cpu().numpy()[:, :D]
        rows = rows_visited(nodes, alen, haschild[(Wm + i) % pool])
        alg_bytes += int(rows.sum()) * V * es
        rows_read += int(rows.sum())
        emitted += int((alen + 1).sum())
        accepted += int(alen.sum())
    mean_launch_s = (sum(launch_ms) / K) / 1e3
    achieved_gbs = (alg_bytes / K) / mean_launch_s / 1e9
    peak, peak_kind = measured_peak()

    result = {
        "metric": METRIC, "value": value, "unit": "nodes/s", "n_gpus": world, "steps": K,
        "warmup": Wm, "ms_per_step": elapsed_ms / K, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": w.dtype, "data": "synthetic",
        "config": {
            "workload": w.name if B == w.batch else f"{w.name}@batch{B}", "batch": B, "vocab": V, "nodes_per_seq": N, "max_depth": D,
            "tree": list(w.tree[1]) if w.tree[0] == "levels" else list(w.tree[1:]),
            "logits": f"{w.gen} slope {w.slope} scale {w.scale} rho {w.rho}",
            "temperature": w.temperature, "mode": args.mode, "z_rule": args.z_rule,
            "proxy_denominator": args.proxy_denominator, "fill": args.fill, "draft": args.draft,
            "parallelism": f"replicas{world}" if world > 1 else "single",
            "launch": {k: plan[k] for k in ("kernel_name", "cluster_size", "block_threads",
                                            "smem_bytes", "slice_elems", "uses_tma",
                                            "vector_loads",
                                            "active_clusters")}
                      | {"kernel_source_digest": kernel_source_digest()},
            "l2": f"rotating pool of {pool} input sets ({set_bytes / 1e9:.2f} GB each) "
                  f"between steps; each step's visited rows exceed L2 together",
        },
        "roofline": {"bound": "hbm", "achieved": achieved_gbs, "peak": peak, "unit": "GB/s",
                     "frac": achieved_gbs / peak,
                     "traffic": profiled_traffic(plan["kernel_name"], w.name, alg_bytes / K),
                     "peak_kind": peak_kind, "frac_of_8tbs": achieved_gbs / NOMINAL_HBM_GBS,
                     "alg_bytes_per_launch": alg_bytes / K,
                     "mean_launch_us": mean_launch_s * 1e6,
                     "median_launch_us": statistics.median(launch_ms) * 1e3},
        "tokens_per_s": sum_over_ranks(float(emitted)) / (elapsed_ms / 1e3),
        # nodes whose rows were read (the root and every accepted node): one
        # emitted token each, so equal to tokens_per_s
        "visited_nodes_per_s": sum_over_ranks(float(emitted)) / (elapsed_ms / 1e3),
        "rows_read_per_s": sum_over_ranks(float(rows_read)) / (elapsed_ms / 1e3),
        "mean_accept_len": accepted / (K * B),
        "gpu_launches": K,
        "wall_s": wall,
    }
    if clk:
        result["clocks"] = clk

    # ---- end to end through the public API with host buffers
    if not args.no_e2e:
        s0 = sets[0]
        host = {k: s0[k].cpu().pin_memory() for k in ("target", "draft", "cand")}
        host["parents"] = s0["parents"].cpu().pin_memory()
        dbuf = {k: torch.empty_like(s0[k]) for k in ("target", "draft", "cand", "parents")}
        h_tok = torch.empty((B, D + 1), dtype=torch.int32).pin_memory()
        h_len = torch.empty((B,), dtype=torch.int32).pin_memory()
        d_tok = torch.empty((B, D + 1), dtype=torch.int32, device=dev)
        d_len = torch.empty((B,), dtype=torch.int32, device=dev)
        # drafting: the kernel writes the drafted children here (the same work
        # as the timed steps)
        e2e_kw = {"out_candidates": torch.empty((B, N), dtype=torch.int32, device=dev)} \
            if args.draft else {}
        h2d = sum(t.numel() * t.element_size() for t in host.values())
        d2h = h_tok.numel() * 4 + h_len.numel() * 4
        E = max(1, args.e2e_steps)

        def e2e_step(i):
            for k in dbuf:
                dbuf[k].copy_(host[k], non_blocking=True)
            rs.verify(dbuf["target"], dbuf["draft"], dbuf["parents"], dbuf["cand"],
                      w.temperature, args.seed + i, out_tokens=d_tok, out_accept_len=d_len,
                      max_depth=D, mode=mode, stream=stream, kernel=kernel, z_rule=z_rule,
                      proxy_denominator=args.proxy_denominator, fill=fill, **e2e_kw)
            h_tok.copy_(d_tok, non_blocking=True)
            h_len.copy_(d_len, non_blocking=True)

        e2e_step(0)
        torch.cuda.synchronize()
        barrier()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        for i in range(E):
            e2e_step(i + 1)
        e1.record(stream)
        torch.cuda.synchronize()
        barrier()
        e_ms = max_over_ranks(e0.elapsed_time(e1))
        result["e2e"] = {"value": sum_over_ranks(float(E * B * N)) / (e_ms / 1e3),
                         "unit": "nodes/s", "h2d_bytes_per_step": h2d,
                         "d2h_bytes_per_step": d2h, "steps": E}
        del host, dbuf

    # ---- the first step's call again, with the outputs the parity sample
    # compares (accepted node ids and rejection counts; not timed)
    gpu_ref = None
    if not args.no_cpu_baseline and world == 1:
        s0 = sets[0]
        ref = {"tokens": torch.empty((B, D + 1), dtype=torch.int32, device=dev),
               "accept_len": torch.empty((B,), dtype=torch.int32, device=dev),
               "nodes": torch.empty((B, max(D, 1)), dtype=torch.int32, device=dev),
               "rejects": torch.empty((B,), dtype=torch.int32, device=dev)}
        rs.verify(s0["target"], s0["draft"], s0["parents"], None if args.draft else s0["cand"],
                  w.temperature, args.seed, out_tokens=ref["tokens"],
                  out_accept_len=ref["accept_len"], out_nodes=ref["nodes"],
                  out_rejects=ref["rejects"], stream=stream, out_candidates=drafted, **kw)
        torch.cuda.synchronize()
        gpu_ref = {k: v.cpu().numpy() for k, v in ref.items()}

    # ---- the oracle as it stands on the host cores (rank 0, N = 1 only)
    result = _finish_cpu(result, args, sets, w, mode, world, dev, gpu_ref)
    if rank == 0:
        print(json.dumps(result), flush=True)
    if dist is not None:
        dist.destroy_process_group()
    return 0


def _host_logits(t):
    import torch
    if t.dtype == torch.bfloat16:
        return t.contiguous().view(torch.int16).cpu().numpy().view(np.uint16)
    return t.contiguous().cpu().numpy()


def _finish_cpu(result, args, sets, w, mode, world, dev, gpu_ref=None):
    if args.no_cpu_baseline or world != 1:
        return result
    import torch
    import oracle
    s0 = sets[0]
    S = max(1, min(args.cpu_seqs, int(s0["cand"].shape[0])))
    idx = torch.arange(S, device=dev)
    th = _host_logits(s0["target"].index_select(0, idx))
    dh = _host_logits(s0["draft"].index_select(0, idx))
    ch = s0["cand"].index_select(0, idx).cpu().numpy()
    omode = oracle.MODE_SPECINFER if mode == 1 else oracle.MODE_RESISPEC
    pa = s0["parents_np"][:S] if w.per_sequence_tree else s0["parents_np"]
    rate, threads, sample, one = cpu_oracle_rate(w, th, dh, pa, ch,
                                                 np.arange(S, dtype=np.int32), omode,
                                                 args.cpu_seconds, args.seed, oracle_variant(args))
    result["cpu_baseline"] = {"value": rate, "unit": "nodes/s", "cores": threads,
                              "kind": "oracle", "sample": sample, "one_thread_value": one,
                              "cpu_model": cpu_model(), "nproc": os.cpu_count()}
    # parity of this run's GPU outputs on the same sequences and seed (the
    # first S sequences of input set 0, seed args.seed: the first warm-up
    # step's call, repeated with the optional outputs)
    if gpu_ref is not None:
        variant = oracle_variant(args)
        o = oracle.verify(th, dh, pa, ch, w.temperature, args.seed, mode=omode,
                          max_depth=w.max_depth, seq_ids=np.arange(S, dtype=np.int32),
                          **variant)
        if variant.get("draft_children"):
            o["sample_margin"] = np.minimum(o["sample_margin"], o["draft_margin"])
        g = {k: v[:S] for k, v in gpu_ref.items()}
        result["parity_sample"] = parity_sample(g, o)
    return result


def main(argv=None):
    args = parse_args(argv)
    if args.impl == "reference":
        return run_reference(args)
    return run_ours(args)


if __name__ == "__main__":
    sys.exit(main())
