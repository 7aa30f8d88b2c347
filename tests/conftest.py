import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)
TESTS = os.path.dirname(os.path.abspath(__file__))
if TESTS not in sys.path:
    sys.path.insert(0, TESTS)


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a CUDA GPU (GB300, sm_103a) and the built library")


def pytest_terminal_summary(terminalreporter):
    """Totals of the GPU parity checks: the entries excluded as near ties or
    near the threshold (and how many of those actually differ), the
    library's own counters, the worst output errors and the largest output
    magnitude met."""
    mod = sys.modules.get("gpu_harness")
    if mod is None or not getattr(mod, "REPORTS", None):
        return
    tr = terminalreporter
    tot = dict(tokens=0, near_route=0, near_route_logit=0, near_route_diff=0, lib_route=0, branches=0,
               near_score=0, near_score_diff=0, lib_score=0, widened=0)
    worst_rel, worst_abs, max_out = 0.0, 0.0, 0.0
    for _, r in mod.REPORTS:
        tot["tokens"] += r.tokens_routed
        tot["near_route"] += r.near_route
        tot["near_route_logit"] += r.near_route_logit
        tot["near_route_diff"] += r.near_route_diff
        tot["lib_route"] += r.lib_near_route
        tot["branches"] += r.branches
        tot["near_score"] += r.near_score
        tot["near_score_diff"] += r.near_score_diff
        tot["lib_score"] += r.lib_near_score
        tot["widened"] += r.widened
        worst_rel, worst_abs, max_out = max(worst_rel, r.max_rel_l2), max(worst_abs, r.max_abs), max(max_out, r.max_out)
    tr.write_sep("-", "GPU parity: excluded entries and output errors")
    tr.write_line(f"trajectories checked: {len(mod.REPORTS)}; tokens routed {tot['tokens']}, branches {tot['branches']}")
    tr.write_line(f"near-tie tokens excluded (gap < 1e-5 cond): {tot['near_route']} "
                  f"({tot['near_route'] / max(tot['tokens'], 1):.2e}); under the |logit| window: "
                  f"{tot['near_route_logit']}; library counter: {tot['lib_route']}; of the excluded, ids differ on "
                  f"{tot['near_route_diff']}")
    tr.write_line(f"near-threshold branches excluded (|s - tau| < 1e-5 |tau|): {tot['near_score']} "
                  f"({tot['near_score'] / max(tot['branches'], 1):.2e}); library counter: {tot['lib_score']}; "
                  f"decisions differ on {tot['near_score_diff']}")
    tr.write_line(f"worst output rel L2 {worst_rel:.2e}, worst max abs {worst_abs:.2e}, largest |output| "
                  f"{max_out:.1f}, elements whose bound exceeds 5e-2 {tot['widened']}")
    for name, r in mod.REPORTS:
        if r.near_route or r.near_score:
            tr.write_line(f"  {name}: {r.summary()}")
