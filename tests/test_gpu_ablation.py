"""The granularity / score-signal ablation driver on the GPU path (small fp32 workload).

Token-level decisions recompute a superset of the branch-level recompute set
(the OR rule, pinned on the oracle), so at the same tau0 they never reuse
more; the calibration reaches a reachable target; no-reuse runs agree.
"""
import math

import pytest

pytestmark = pytest.mark.gpu


def test_ablation_trajectory_rules():
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    from paper_2606_15615_gb300 import ablation as A
    from paper_2606_15615_gb300 import workloads as W
    wl = W.WORKLOADS["moe_d384_e8_k2_f1536_t512_l1_f32"]
    tr = A._Trajectory(wl, 6, refresh_period=0)
    branch, token = tr.stack(7, 0), tr.stack(7, 1)
    _, _, dense_b = tr.run(branch, -math.inf, True)
    _, _, dense_t = tr.run(token, -math.inf, True)
    for a, b in zip(dense_b, dense_t):
        assert A.rel_l2(a, b) == 0.0  # nothing reused: both rules recompute everything
    for tau0 in (0.4, 0.7, 1.0):
        rb = tr.run(branch, tau0, False)[0]
        rt = tr.run(token, tau0, False)[0]
        assert rt <= rb + 1e-12, (tau0, rt, rb)
    tau0 = tr.calibrate(branch, 0.3)
    r, _, outs = tr.run(branch, tau0, True)
    assert abs(r - 0.3) < 0.05
    errs = [A.rel_l2(o, d) for o, d in zip(outs, dense_b)]
    assert all(math.isfinite(e) for e in errs) and max(errs) > 0.0
    for st in (branch, token):
        st.close()
