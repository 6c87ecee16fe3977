"""Synthetic replication of the paper's verification diagnostics on the GPU
path.

* Acceptance by candidate position (Sec. 3, "The Decay of Acceptance
  Probability"): for a single position with k i.i.d. candidates, the rate
  at which candidate i is accepted given that candidates 1..i-1 were
  rejected.  SpecInfer's residual drifts away from the draft, so the rate
  falls after the first candidate; ResiSpec's shaping is meant to hold it.
* Scaling efficiency (App., "Scaling Inefficiency of Multi-Candidate
  Schemes"): with the depth fixed, the expected accepted length EAL
  (emitted tokens per step: accepted candidates + 1) for N candidates per
  position, its marginal gain and eta = delta EAL / delta N.
* Runtime breakdown (Sec. 6, "Computational Overhead"): the share of each
  verification phase in the kernel's own cycle counters (budgeting is part
  of the accept tests, redistribution is the rejection passes; the proxy is
  never materialised).

The statistics are functions of the verification outputs only, so the same
functions applied to the oracle's outputs on the same inputs must agree
(the GPU tests check it).  ``python -m paper_2608_24411_gb300.diagnostics``
runs all three on synthetic inputs on cuda:0 and prints one JSON object.
The inputs stand in for the paper's models and datasets (Llama-2 / CNN-DM),
which are not used here.
"""
from __future__ import annotations

import json
import sys

import numpy as np


def accepted_position(accept_len, nodes, k: int) -> np.ndarray:
    """For single-position trees (node i = candidate i + 1 of the root):
    the 0-based position of the accepted candidate, k when all k were
    rejected, -1 for a sequence with a data error."""
    a = np.asarray(accept_len)
    n = np.asarray(nodes)
    pos = np.where(a >= 1, n[:, 0] if n.ndim == 2 and n.shape[1] else -1, k)
    return np.where(a < 0, -1, pos).astype(np.int64)


def position_rates(pos, k: int):
    """(reached[i], accepted[i], rate[i]) for i < k: sequences that tested
    candidate i, those that accepted it, and their ratio."""
    pos = np.asarray(pos)
    pos = pos[pos >= 0]
    reached = np.array([(pos >= i).sum() for i in range(k)], dtype=np.int64)
    accepted = np.array([(pos == i).sum() for i in range(k)], dtype=np.int64)
    rate = np.divide(accepted, reached, out=np.zeros(k), where=reached > 0)
    return reached, accepted, rate


def scaling_table(eal_by_n: dict):
    """Rows (N, EAL, delta EAL, eta) in ascending N; eta = delta EAL / delta N
    against the previous row (None for the first)."""
    rows, prev = [], None
    for n in sorted(eal_by_n):
        e = float(eal_by_n[n])
        if prev is None:
            rows.append((n, e, None, None))
        else:
            d = e - prev[1]
            rows.append((n, e, d, d / (n - prev[0])))
        prev = (n, e)
    return rows


def phase_shares(cycles) -> dict:
    """Share of each phase in the summed cycles of all sequences."""
    from . import PHASES
    c = np.asarray(cycles, dtype=np.float64).sum(axis=0)
    tot = c.sum()
    return {name: (float(c[i] / tot) if tot > 0 else 0.0) for i, name in enumerate(PHASES)}


# ------------------------------------------------------------------ runs


def _verify(inp, mode, seed, **kw):
    import torch
    from . import verify
    B = int(inp["cand"].shape[0])
    D = int(inp["max_depth"])
    nodes = torch.full((B, max(D, 1)), -1, dtype=torch.int32, device=inp["target"].device)
    toks, alen = verify(inp["target"], inp["draft"], inp["parents"], inp["cand"],
                        inp["temperature"], seed, max_depth=D, mode=mode, out_nodes=nodes, **kw)
    torch.cuda.synchronize()
    return alen.cpu().numpy(), nodes.cpu().numpy()


def run(device="cuda:0", batch=4096, seed=0) -> dict:
    from . import MODE_RESISPEC, MODE_SPECINFER, PHASES
    from . import workloads as W
    import torch

    out = {"inputs": "synthetic (zipf logits, V = 32000 bf16, T = 1); "
                     "stand-ins for the paper's models and datasets"}
    modes = {"resispec": MODE_RESISPEC, "specinfer": MODE_SPECINFER}
    # acceptance by candidate position: one position, k = 8 candidates
    k = 8
    w = W.Workload(name="decay", batch=batch, vocab=32000, dtype="bf16", gen="zipf", scale=3.0,
                   slope=1.1, rho=0.8, temperature=1.0, tree=("single", k), steps=1)
    inp = W.make_inputs_torch(w, seed, device)
    decay = {}
    for name, mode in modes.items():
        alen, nodes = _verify(inp, mode, seed + 1)
        reached, accepted, rate = position_rates(accepted_position(alen, nodes, k), k)
        decay[name] = {"rate": [round(float(r), 4) for r in rate],
                       "reached": reached.tolist()}
    out["acceptance_by_position"] = decay
    del inp
    # scaling efficiency: chain of depth 4, N candidates per position
    eta = {}
    for name, mode in modes.items():
        eal = {}
        for n in (1, 2, 4, 8):
            w = W.Workload(name="eta", batch=batch // 2, vocab=32000, dtype="bf16", gen="zipf",
                           scale=3.0, slope=1.1, rho=0.8, temperature=1.0,
                           tree=("chain", 4, n), steps=1)
            inp = W.make_inputs_torch(w, seed + n, device)
            alen, _ = _verify(inp, mode, seed + 10 + n)
            eal[n] = float((alen[alen >= 0] + 1).mean())
            del inp
        eta[name] = [{"N": n, "EAL": round(e, 4),
                      "dEAL": None if d is None else round(d, 4),
                      "eta": None if h is None else round(h, 4)}
                     for n, e, d, h in scaling_table(eal)]
    out["scaling_efficiency_depth4"] = eta
    # runtime breakdown on the binary depth-5 tree at V = 151936 fp32
    w = W.WORKLOADS["binary5-v151936-b64"]
    inp = W.make_inputs_torch(w, seed, device)
    phases = {}
    for name, mode in modes.items():
        cyc = torch.zeros((w.batch, len(PHASES)), dtype=torch.int64, device=device)
        _verify(inp, mode, seed + 2, out_phase=cyc)
        phases[name] = {p: round(v, 4) for p, v in phase_shares(cyc.cpu().numpy()).items()}
    out["phase_shares_binary5"] = phases
    torch.cuda.empty_cache()
    return out


if __name__ == "__main__":
    import os
    sys.path.insert(0, os.path.dirname(os.path.dirname(os.path.abspath(__file__))))
    print(json.dumps(run()), flush=True)
