"""Multi-rank host logic of bench.py on CPU: one process per rank (gloo,
world size 2), as the replicas run launches one per GPU.  The path has no
data exchange between ranks; only the timing barrier and the reductions
that form the whole-job number cross ranks."""
import json
import os
import socket
import subprocess
import sys

import numpy as np
import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)

import bench  # noqa: E402


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, out_dir):
    import torch
    import torch.distributed as dist
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    g = bench.RankGroup(dist, torch.device("cpu"))
    g.barrier()
    # rank r processed 100 (r + 1) units in 10 (r + 1) ms
    value, slowest = bench.whole_job_rate(g, 100.0 * (rank + 1), 10.0 * (rank + 1))
    res = {"max": g.max(float(rank) + 0.5), "sum": g.sum(float(rank) + 1.0), "value": value,
           "slowest": slowest, "seeds": [bench.replica_seed(1234, rank, i) for i in range(3)]}
    g.barrier()
    dist.destroy_process_group()
    with open(os.path.join(out_dir, f"rank{rank}.json"), "w") as f:
        json.dump(res, f)


def test_rank_group_single_process():
    g = bench.RankGroup()
    g.barrier()
    assert g.max(3.0) == 3.0 and g.sum(2.5) == 2.5
    value, slowest = bench.whole_job_rate(g, 500.0, 250.0)
    assert slowest == 250.0 and value == pytest.approx(2000.0)


def test_rank_group_gloo_world2(tmp_path):
    torch = pytest.importorskip("torch")
    import torch.multiprocessing as mp
    mp.start_processes(_worker, args=(2, _free_port(), str(tmp_path)), nprocs=2,
                       start_method="spawn")
    r = [json.load(open(tmp_path / f"rank{i}.json")) for i in range(2)]
    for x in r:
        assert x["max"] == 1.5 and x["sum"] == 3.0
        # 300 units over the slowest rank's 20 ms
        assert x["slowest"] == 20.0 and x["value"] == pytest.approx(300.0 / 0.020)
    # every replica verifies its own inputs
    assert not set(r[0]["seeds"]) & set(r[1]["seeds"])


def test_reference_arm_under_torchrun_world2(tmp_path):
    """`bench.py --impl reference` launched the way the driver launches N > 1
    runs: rank 0 alone times the oracle and prints one line; rank 1 exits 0."""
    pytest.importorskip("torch")
    import oracle
    oracle.build()
    cmd = [sys.executable, "-m", "torch.distributed.run", "--nnodes=1", "--nproc-per-node", "2",
           "--master-addr", "127.0.0.1", "--master-port", str(_free_port()),
           os.path.join(ROOT, "bench.py"), "--impl", "reference", "--gpus", "2", "--steps", "2",
           "--warmup", "1", "--cpu-seqs", "4", "--workload", "tiny-chain-v64"]
    p = subprocess.run(cmd, cwd=ROOT, capture_output=True, text=True, timeout=300)
    assert p.returncode == 0, p.stderr[-2000:]
    lines = [l for l in p.stdout.splitlines() if l.startswith("{")]
    assert len(lines) == 1, p.stdout
    d = json.loads(lines[0])
    assert d["impl"] == "reference" and d["n_gpus"] == 2 and d["value"] > 0
    assert d["e2e"]["h2d_bytes_per_step"] == 0 and d["cpu_baseline"]["kind"] == "oracle"


def test_rows_visited_per_sequence_trees():
    import bench
    # sequence 0: root -> node 0 (leaf); sequence 1: root -> node 1 -> node 2 (leaf)
    parents = np.array([[-1, -1, 1], [-1, -1, 1]], np.int32)
    hc = bench.has_children(parents)
    assert hc.shape == (2, 4) and hc[0, 0] and hc[0, 2] and not hc[0, 1] and not hc[0, 3]
    nodes = np.array([[0, -1], [1, 2]], np.int32)
    alen = np.array([1, 2], np.int32)
    # root (2 rows) + leaf 0 (1 row); root (2) + node 1 (2) + leaf 2 (1)
    np.testing.assert_array_equal(bench.rows_visited(nodes, alen, hc), [3, 5])
    np.testing.assert_array_equal(bench.rows_visited(nodes, alen, bench.has_children(parents[0])),
                                  [3, 5])


def test_reference_arm_times_the_variant_it_is_asked_for():
    """The oracle legs verify with the same rule as the measured run."""
    import argparse
    import bench
    ns = argparse.Namespace(z_rule="applied", proxy_denominator=True, fill="level", draft=False)
    assert bench.oracle_variant(ns) == dict(z_rule=1, denom_update=True, fill=1,
                                            draft_children=False)
    ns = argparse.Namespace(z_rule="alg1", proxy_denominator=False, fill="capacity", draft=True)
    assert bench.oracle_variant(ns) == dict(z_rule=0, denom_update=False, fill=0,
                                            draft_children=True)
    cmd = [sys.executable, os.path.join(ROOT, "bench.py"), "--impl", "reference", "--steps", "1",
           "--warmup", "0", "--cpu-seqs", "4", "--workload", "tiny-chain-v64", "--fill", "level",
           "--proxy-denominator"]
    p = subprocess.run(cmd, cwd=ROOT, capture_output=True, text=True, timeout=300)
    assert p.returncode == 0, p.stderr[-2000:]
    d = json.loads([l for l in p.stdout.splitlines() if l.startswith("{")][-1])
    assert d["config"]["fill"] == "level" and d["config"]["proxy_denominator"] is True


@pytest.mark.parametrize("wl", ["tiny-chain-v64", "dyntree60-v32000"])
def test_cpu_oracle_rate_on_host_inputs(wl):
    """The CPU-baseline leg of the GPU arm, on host copies of a workload
    (one shared tree, and a tree per sequence)."""
    import bench
    import oracle
    from paper_2608_24411_gb300 import workloads as W
    w = W.WORKLOADS[wl]
    inp = W.make_inputs_np(w, seed=0, batch=4)
    rate, threads, sample, one = bench.cpu_oracle_rate(
        w, inp["target"], inp["draft"], inp["parents"], inp["cand"],
        np.arange(4, dtype=np.int32), oracle.MODE_RESISPEC, 0.05, 1, {"fill": 1})
    assert rate > 0 and one > 0 and 1 <= threads <= 4 and "verified nodes" in sample
    assert isinstance(bench.cpu_model(), str)


def test_parity_sample_counts_ties_and_mismatches():
    """bench.parity_sample on hand-made outputs: a difference inside the tie
    band is counted as such, one outside it separately, and the near-tie
    counts follow the oracle's margins level by level."""
    o = {"accept_len": np.array([1, 2, 0, 1]), "tokens": np.array([[5, 7, -1], [5, 6, 9], [3, -1, -1], [4, 4, -1]]),
         "nodes": np.array([[0, -1], [0, 2], [-1, -1], [1, -1]]), "rejects": np.array([0, 1, 2, 1]),
         "accept_margin": np.array([0.3, 5e-6, 0.2, 2e-8]), "sample_margin": np.array([0.1, 0.2, 5e-7, 0.4])}
    g = {k: np.array(v, copy=True) for k, v in o.items() if k in ("accept_len", "tokens", "nodes", "rejects")}
    g["tokens"][1, 2] = 8      # sequence 1 differs: accept margin 5e-6 is a near tie
    g["tokens"][0, 1] = 3      # sequence 0 differs with no near tie
    r = bench.parity_sample(g, o)
    assert r["sequences"] == 4
    assert r["mismatch_in_ties"] == 1 and r["mismatch_outside_ties"] == 1
    assert r["near_tie"]["accept<=1e-05"] == 2 and r["near_tie"]["accept<=1e-06"] == 1
    assert r["near_tie"]["accept<=1e-07"] == 1 and r["near_tie"]["sample<=1e-06"] == 1
    assert r["near_tie"]["sample<=1e-07"] == 0
