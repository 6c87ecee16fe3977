import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a CUDA GPU (sm_103a) and the built library")
    config.addinivalue_line("markers", "slow: long-running statistical check")


def pytest_collection_modifyitems(config, items):
    # GPU tests need the device; skip them cleanly when none is present.
    try:
        import torch
        has_gpu = torch.cuda.is_available()
    except Exception:  # pragma: no cover
        has_gpu = False
    if has_gpu:
        return
    skip = pytest.mark.skip(reason="no CUDA device")
    for it in items:
        if "gpu" in it.keywords:
            it.add_marker(skip)


@pytest.fixture(scope="session")
def oracle_lib():
    import oracle
    oracle.build()
    return oracle.load()


def pytest_terminal_summary(terminalreporter, exitstatus, config):
    """Near-tie report of the GPU parity comparisons that ran: per test, the
    sequences compared, how many sit within 1e-5 / 1e-6 / 1e-7 of an accept
    or final-draw tie (oracle margins, fp64), how many of those differ from
    the oracle, and the worst residual error."""
    parity = sys.modules.get("tests.parity")
    if parity is None or not parity.REPORTS:
        return
    agg = {}
    for r in parity.REPORTS:
        a = agg.setdefault(r["label"], {"calls": 0, "sequences": 0, "mismatch_in_ties": 0,
                                        "near_tie": {}, "dist_maxabs": 0.0, "dist_l1": 0.0})
        a["calls"] += 1
        a["sequences"] += r["sequences"]
        a["mismatch_in_ties"] += r["mismatch_in_ties"]
        for k, v in r["near_tie"].items():
            a["near_tie"][k] = a["near_tie"].get(k, 0) + v
        a["dist_maxabs"] = max(a["dist_maxabs"], r["dist_maxabs"])
        a["dist_l1"] = max(a["dist_l1"], r["dist_l1"])
    tr = terminalreporter
    tr.section("near-tie report: GPU vs oracle (fp64 accept decisions)")
    keys = [f"{w}<={t:g}" for t in parity.TIE_LEVELS for w in ("accept", "sample")]
    tr.write_line("sequences  " + "  ".join(keys) + "  mismatch_in_ties  dist_maxabs  dist_l1  test")
    tot = {"sequences": 0, "mismatch_in_ties": 0, **{k: 0 for k in keys}}
    for label, a in agg.items():
        tot["sequences"] += a["sequences"]
        tot["mismatch_in_ties"] += a["mismatch_in_ties"]
        for k in keys:
            tot[k] += a["near_tie"].get(k, 0)
        tr.write_line(f"{a['sequences']:9d}  " + "  ".join(f"{a['near_tie'].get(k, 0):>{len(k)}d}"
                                                          for k in keys)
                      + f"  {a['mismatch_in_ties']:16d}  {a['dist_maxabs']:11.2e}  "
                        f"{a['dist_l1']:7.2e}  {label}")
    tr.write_line(f"{tot['sequences']:9d}  " + "  ".join(f"{tot[k]:>{len(k)}d}" for k in keys)
                  + f"  {tot['mismatch_in_ties']:16d}  (all comparisons; mismatches outside "
                    f"ties: 0, or the test failed)")
