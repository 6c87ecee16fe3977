"""Helpers shared by the GPU parity tests: run the CUDA path and the fp64
oracle on the same seeded inputs and compare them.

Parity rule (the tolerances of the verification hot path):
  * every sequence is compared: accepted tokens, accept length, accepted
    node ids, rejection count and the final token must be bit-exact;
  * a difference is allowed only for a sequence where the oracle saw a near
    tie: an accept test with |u - R(x)/q(x)| <= 1e-5, or a final draw whose
    relative CDF margin is <= 1e-6 (the fp32 distribution the kernel draws
    from carries about 1e-7 relative rounding per probability, so a margin
    below that bound can legitimately fall either way); such differences
    are counted and reported;
  * the distribution of the final draw (for every sequence whose path
    matches) agrees within 1e-6 max-abs and 1e-5 L1 per row, and the GPU
    row sums to 1 within 1e-6, in both modes (the kernel evaluates the
    SpecInfer residual (p - C q)_+ / N with double-float sums and
    exponentials where the residual's conditioning 1 / N demands them).
    Rows whose test denominator is the proxy (the EAGLE-integration
    variant) add, token by token, the oracle's first-order bound of the
    error of an fp32 evaluation of the chain ("dist_err"): the proxy
    K = R - r cancels on tokens next to the level and a later small budget
    divides it (0 for every other row).
"""
import os

import numpy as np

import oracle
import paper_2608_24411_gb300 as rs

ACCEPT_TIE = 1e-5
SAMPLE_TIE = 1e-6
DIST_MAXABS = 1e-6
DIST_L1 = 1e-5


def to_host_logits(t):
    """torch tensor (float32 or bfloat16) -> numpy array the oracle accepts."""
    import torch
    if t.dtype == torch.bfloat16:
        return t.contiguous().view(torch.int16).cpu().numpy().view(np.uint16)
    return t.contiguous().cpu().numpy()


def to_device(arr, device="cuda"):
    import torch
    if arr.dtype == np.uint16:
        return torch.from_numpy(arr.view(np.int16)).to(device).view(torch.bfloat16)
    return torch.from_numpy(np.ascontiguousarray(arr)).to(device)


def run_gpu(target, draft, parents, cand, T, seed, max_depth, mode=rs.MODE_RESISPEC,
            want_dist=True, **kw):
    """target/draft/parents/cand: torch CUDA tensors."""
    import torch
    B = (cand if cand is not None else kw["out_candidates"]).shape[0]
    V = target.shape[-1]
    dev = target.device
    out = {
        "nodes": torch.full((B, max(max_depth, 1)), -7, dtype=torch.int32, device=dev),
        "rejects": torch.full((B,), -7, dtype=torch.int32, device=dev),
        "status": torch.zeros((1,), dtype=torch.int32, device=dev),
    }
    if want_dist:
        out["dist"] = torch.full((B, V), -1.0, dtype=torch.float32, device=dev)
    toks, alen = rs.verify(target, draft, parents, cand, T, seed, max_depth=max_depth,
                           mode=mode, out_nodes=out["nodes"], out_dist=out.get("dist"),
                           out_rejects=out["rejects"], status=out["status"], **kw)
    torch.cuda.synchronize()
    res = {k: v.cpu().numpy() for k, v in out.items()}
    res["tokens"] = toks.cpu().numpy()
    res["accept_len"] = alen.cpu().numpy()
    res["nodes"] = res["nodes"][:, :max_depth]
    return res


def run_oracle(target_h, draft_h, parents_h, cand_h, T, seed, max_depth, mode, seq_ids=None,
               want_dist=True, seq_stride=None, z_rule=0, denom_update=False, fill=0):
    """The oracle on the same inputs, taking every accept decision as the
    paper writes it: u < R(x)/D(x) in fp64."""
    return oracle.verify(target_h, draft_h, parents_h, cand_h, T, seed, mode=mode,
                         decide_fp64=True,
                         max_depth=max_depth, seq_ids=seq_ids, want_dist=want_dist,
                         seq_stride=seq_stride, z_rule=z_rule, denom_update=denom_update,
                         fill=fill, want_dist_err=want_dist and denom_update)


TIE_LEVELS = (1e-5, 1e-6, 1e-7)

# Every comparison made in this process, for the session's near-tie report
# (printed by the terminal-summary hook in conftest.py).
REPORTS = []


def near_tie_counts(o, idx=None):
    """Sequences whose accept margin |u - R(x)/D(x)| (any test of the walk)
    or whose final-draw CDF margin (relative) is at or below each level of
    TIE_LEVELS, from the oracle's fp64 margins."""
    am, sm = o["accept_margin"], o["sample_margin"]
    if idx is not None:
        am, sm = am[idx], sm[idx]
    out = {}
    for t in TIE_LEVELS:
        out[f"accept<={t:g}"] = int((am <= t).sum())
        out[f"sample<={t:g}"] = int((sm <= t).sum())
    return out


def compare(g, o, rows=None, check_dist=True, label=None):
    """Compare GPU outputs g (rows `rows` of the batch, or all) with oracle
    outputs o under the parity rule above.  Returns a report dict: the
    sequences compared, the near-tie counts at 1e-5 / 1e-6 / 1e-7, the
    sequences that differ inside the tie band ("mismatch_in_ties"; those
    outside it fail the comparison), and the worst residual errors."""
    idx = np.arange(len(o["accept_len"])) if rows is None else np.asarray(rows)
    sel = lambda a: a[idx]
    near = (o["accept_margin"] <= ACCEPT_TIE) | (o["sample_margin"] <= SAMPLE_TIE)
    errs = (o["status"] & ~oracle.INFO_DEGENERATE) != 0
    gl, ol = sel(g["accept_len"]), o["accept_len"]
    gt, ot = sel(g["tokens"]), o["tokens"]
    same_path = gl == ol
    if "nodes" in g and o["nodes"].shape[1]:
        gn = sel(g["nodes"])[:, : o["nodes"].shape[1]]
        same_path &= (gn == o["nodes"]).all(axis=1)
    if "rejects" in g:
        same_path &= errs | (sel(g["rejects"]) == o["rejects"])
    differs = ~same_path | (gt != ot).any(axis=1)
    bad = np.nonzero(differs & ~near)[0]
    assert bad.size == 0, (f"{bad.size} sequences differ without a near tie, e.g. {bad[:5]}: "
                           f"gpu len {gl[bad[:5]]} tokens {gt[bad[:3]]}; "
                           f"oracle len {ol[bad[:5]]} tokens {ot[bad[:3]]}; "
                           f"margins {o['accept_margin'][bad[:5]]} {o['sample_margin'][bad[:5]]}")
    rep = {"label": label or os.environ.get("PYTEST_CURRENT_TEST", "").split(" ")[0],
           "sequences": int(len(idx)), "near_tie": near_tie_counts(o),
           "mismatch_in_ties": int((differs & near).sum()), "mismatch_outside_ties": 0,
           "dist_rows": 0, "dist_maxabs": 0.0, "dist_l1": 0.0}
    if check_dist and "dist" in g and "dist" in o:
        gd = sel(g["dist"]).astype(np.float64)
        ok = same_path & ~errs
        if ok.any():
            diff = np.abs(gd[ok] - o["dist"][ok])
            bar = o["dist_err"][ok] if "dist_err" in o else np.zeros_like(diff)
            worst = (diff - bar).max()
            l1 = np.maximum(diff - bar, 0).sum(axis=1)
            rep.update(dist_rows=int(ok.sum()), dist_maxabs=float(worst), dist_l1=float(l1.max()),
                       dist_maxabs_raw=float(diff.max()),
                       dist_l1_raw=float(diff.sum(axis=1).max()),
                       cond_max=float(o["cond"][ok].max()))
            assert worst <= DIST_MAXABS, f"dist max-abs {worst:.3e} beyond the error bound"
            assert l1.max() <= DIST_L1, f"dist L1 {l1.max():.3e}"
            sums = gd[ok].sum(axis=1)
            assert np.abs(sums - 1).max() <= 1e-6, f"residual sum off by {np.abs(sums - 1).max():.3e}"
            assert (gd[ok] >= 0).all()
    REPORTS.append(rep)
    print(f"parity {rep['label']}: {rep['sequences']} sequences, near ties {rep['near_tie']}, "
          f"mismatches in ties {rep['mismatch_in_ties']}, residual rows {rep['dist_rows']} "
          f"(max-abs {rep['dist_maxabs']:.2e}, L1 {rep['dist_l1']:.2e}; unscaled max-abs "
          f"{rep.get('dist_maxabs_raw', 0.0):.2e}, L1 {rep.get('dist_l1_raw', 0.0):.2e}, "
          f"largest 1/prod S {rep.get('cond_max', 1.0):.3g})")
    return rep
