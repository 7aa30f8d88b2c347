"""Granularity and score-signal ablation on synthetic trajectories.

Runs the layer stack of a workload through a denoising trajectory under
several decision rules and reports, at matched reuse ratios, how far the
stack output drifts from the no-reuse output:

* branch-level decisions with the full Eq. 9 score (MoECa),
* token-level decisions (Sec. 3): a token's branches share one decision,
* branch-level decisions with each subset of the score terms w, lambda1
  Delta and lambda2 o (the signal ablation of Table 5).

For every rule and target reuse ratio, tau0 is found by bisection on the
GPU path, so that the reused fraction of routed branches over the cache
steps is as close as possible to the target.  Error is the relative L2
distance of the stack output from the no-reuse output (tau0 = -inf, every
branch recomputed), averaged over the cache steps, with the worst step
alongside.  The trajectory's inputs come from the workload generator, not
from a sampler, so the error does not feed back into later inputs.

Usage:  python -m paper_2606_15615_gb300.ablation [--workload NAME] [--steps N]
        [--targets 0.3,0.5,0.7]
Prints one JSON line per (rule, target) and a summary table.
"""
from __future__ import annotations

import argparse
import json
import math

RULES = [
    # name, score_terms, granularity
    ("branch w+D+o (MoECa)", 7, 0),
    ("token w+D+o", 7, 1),
    ("branch w", 1, 0),
    ("branch D", 2, 0),
    ("branch o", 4, 0),
    ("branch w+D", 3, 0),
    ("branch w+o", 5, 0),
    ("branch D+o", 6, 0),
]


class _Trajectory:
    def __init__(self, wl, n_steps: int, refresh_period: int, device: int = 0):
        import torch
        from . import build
        build.build()
        from . import moeca as M
        from . import workloads as W
        self.torch, self.M, self.wl = torch, M, wl
        self.dev = torch.device("cuda", device)
        torch.cuda.set_device(self.dev)
        self.dt = torch.bfloat16 if wl.dtype == "bf16" else torch.float32
        self.weights = [W.make_layer_weights_device(wl, l, self.dev) for l in range(wl.n_layers)]
        self.xs = torch.stack([torch.from_numpy(x) for x in W.trajectory(wl, n_steps)]).to(self.dev).to(self.dt)
        self.n_steps = n_steps
        self.refresh_period = refresh_period

    def stack(self, score_terms: int, granularity: int):
        M, wl = self.M, self.wl
        cfg = M.moeca_config_default(
            n_layers=wl.n_layers, hidden=wl.hidden, ffn=wl.ffn, n_experts=wl.n_experts, top_k=wl.top_k,
            n_shared=wl.n_shared, max_tokens=wl.n_tokens,
            dtype=M.MOECA_BF16 if wl.dtype == "bf16" else M.MOECA_F32, refresh_period=self.refresh_period,
            score_terms=score_terms, granularity=granularity)
        return M.Stack(cfg, self.weights, device=self.dev.index)

    def run(self, st, tau0: float, keep: bool):
        """Whole trajectory; returns (reuse over cache steps, ms per step, outputs or None)."""
        torch, M = self.torch, self.M
        M.moeca_reset(st.handle)
        outs = []
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        st.step(self.xs[0], 0, tau0=tau0)
        torch.cuda.synchronize(self.dev)
        M.moeca_reset_stats(st.handle)
        e0.record()
        for t in range(1, self.n_steps):
            o = st.step(self.xs[t], t, tau0=tau0)
            if keep:
                outs.append(o)
        e1.record()
        torch.cuda.synchronize(self.dev)
        s = M.moeca_get_stats(st.handle)
        reuse = s["reused"] / max(s["branches"], 1)
        return reuse, e0.elapsed_time(e1) / (self.n_steps - 1), (outs if keep else None)

    def calibrate(self, st, target: float):
        lo, hi = 0.0, 4.0
        r_hi = self.run(st, hi, False)[0]
        if r_hi <= target:
            return hi
        best = (hi, r_hi)
        for _ in range(14):
            mid = 0.5 * (lo + hi)
            r = self.run(st, mid, False)[0]
            if abs(r - target) < abs(best[1] - target):
                best = (mid, r)
            if r < target:
                lo = mid
            else:
                hi = mid
        return best[0]


def rel_l2(a, b) -> float:
    a, b = a.float(), b.float()
    return float((a - b).norm() / b.norm().clamp_min(1e-30))


def main(argv=None):
    from . import workloads as W
    ap = argparse.ArgumentParser(description=__doc__.split("\n\n")[0])
    ap.add_argument("--workload", default="moe_d768_e16_k2_f3072_t2048_l12_bf16")
    ap.add_argument("--steps", type=int, default=20)
    ap.add_argument("--targets", default="0.3,0.5,0.7")
    ap.add_argument("--refresh", type=int, default=-1,
                    help="full-computation period N (default: the workload's; the paper uses N = 4)")
    args = ap.parse_args(argv)
    wl = W.WORKLOADS[args.workload]
    targets = [float(t) for t in args.targets.split(",")]
    refresh = wl.refresh_period if args.refresh < 0 else args.refresh
    tr = _Trajectory(wl, args.steps, refresh)
    st = tr.stack(7, 0)
    _, ms_dense, dense = tr.run(st, -math.inf, True)
    dense = [d.clone() for d in dense]
    st.close()
    rows = []
    for name, terms, gran in RULES:
        st = tr.stack(terms, gran)
        for target in targets:
            tau0 = tr.calibrate(st, target)
            reuse, ms, outs = tr.run(st, tau0, True)
            errs = [rel_l2(o, d) for o, d in zip(outs, dense)]
            row = dict(workload=wl.name, refresh_period=refresh, rule=name, score_terms=terms, granularity="token" if gran else "branch",
                       reuse_target=target, reuse=round(reuse, 4), tau0=round(tau0, 5),
                       rel_l2_mean=sum(errs) / len(errs), rel_l2_max=max(errs), ms_per_step=ms,
                       ms_per_step_no_reuse=ms_dense, cache_steps=len(errs))
            rows.append(row)
            print(json.dumps(row), flush=True)
        st.close()
    print(f"\n{'rule':24s} " + " ".join(f"reuse~{t:.1f}: err(mean) reuse" for t in targets))
    for name, _, _ in RULES:
        cells = [r for r in rows if r["rule"] == name]
        print(f"{name:24s} " + " ".join(f"{r['rel_l2_mean']:.3e} {r['reuse']:.3f}      " for r in cells))


if __name__ == "__main__":
    main()
