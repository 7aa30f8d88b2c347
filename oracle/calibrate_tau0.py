"""Calibrate the headline threshold tau0 of a benchmark workload on the oracle.

TEST INFRASTRUCTURE (see moeca_oracle.py): this script calls only the oracle
and the seeded input generators (the weights come from the generator the GPU
benchmark uses, torch's seeded CUDA generator, so it runs on a GPU host; no
kernel of this library runs).  It finds, by bisection, the Eq. 12 base
threshold tau0 at which the oracle reuses the target fraction of routed
branches (reused / routed over the timed steps W .. W + K - 1 of the seeded
trajectory, step 0 a full step), and writes it to
paper_2606_15615_gb300/headline_points.json, which bench.py reads so that
its GPU arm and its reference arm (the oracle) time the same configuration.

  python oracle/calibrate_tau0.py [--workload 2] [--target 0.6] [--warmup 5] [--steps 20]
"""
from __future__ import annotations

import argparse
import json
import os
import sys
import time

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

from oracle import moeca_oracle as O  # noqa: E402
from paper_2606_15615_gb300 import workloads as W  # noqa: E402

OUT = os.path.join(ROOT, "paper_2606_15615_gb300", "headline_points.json")


def layer_weights(wl) -> list:
    """The benchmark's own weights: drawn by torch's seeded CUDA generator
    (workloads.make_layer_weights_device, as the GPU benchmark draws them)
    and copied to host memory as float64 for the oracle."""
    import numpy as np
    import torch
    if not torch.cuda.is_available():
        raise SystemExit("the benchmark weights are drawn by torch's CUDA generator: run this on a GPU host")
    dev = torch.device("cuda", 0)
    out = []
    for l in range(wl.n_layers):
        w = W.make_layer_weights_device(wl, l, dev)
        out.append({k: (None if v is None else v.float().cpu().numpy().astype(np.float64)) for k, v in w.items()})
        del w
    torch.cuda.empty_cache()
    return out


def reuse_at(wl, ws, xs, tau0: float, warmup: int) -> float:
    prm = O.Params(top_k=wl.top_k, tau0=tau0, refresh_period=wl.refresh_period)
    st = O.Stack(ws, prm, wl.hidden, wl.n_experts, wl.n_shared)
    reused = routed = 0
    for t, x in enumerate(xs):
        _, infos = st.step(x, t)
        if t >= warmup:
            for inf in infos:
                reused += int((~inf["recompute"]).sum())
                routed += inf["recompute"].size
    return reused / max(routed, 1)


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--workload", default="2")
    ap.add_argument("--target", type=float, default=0.6)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--steps", type=int, default=20)
    ap.add_argument("--lo", type=float, default=0.5)
    ap.add_argument("--hi", type=float, default=0.8)
    ap.add_argument("--iters", type=int, default=10)
    args = ap.parse_args()
    wl = W.workload(int(args.workload) if args.workload.isdigit() else args.workload)
    t0 = time.time()
    ws = layer_weights(wl)
    xs = list(W.trajectory(wl, args.warmup + args.steps))
    lo, hi = args.lo, args.hi
    r_lo, r_hi = reuse_at(wl, ws, xs, lo, args.warmup), reuse_at(wl, ws, xs, hi, args.warmup)
    if not (r_lo <= args.target <= r_hi):
        raise SystemExit(f"target {args.target} not bracketed: reuse {r_lo:.4f} at {lo}, {r_hi:.4f} at {hi}")
    probes = [(lo, r_lo), (hi, r_hi)]
    for _ in range(args.iters):
        mid = 0.5 * (lo + hi)
        r = reuse_at(wl, ws, xs, mid, args.warmup)
        probes.append((mid, r))
        print(f"tau0 {mid:.6f}: reuse {r:.4f}", flush=True)
        lo, hi = (mid, hi) if r < args.target else (lo, mid)
    tau0, reuse = min(probes, key=lambda p: abs(p[1] - args.target))
    points = {}
    if os.path.exists(OUT):
        with open(OUT) as f:
            points = json.load(f)
    points[wl.name] = {
        "tau0": round(tau0, 6), "reuse_target": args.target, "oracle_reuse": round(reuse, 5),
        "timed_steps": [args.warmup, args.warmup + args.steps - 1],
        "how": (f"bisection on the oracle (oracle/calibrate_tau0.py): reused / routed branches over steps "
                f"{args.warmup}..{args.warmup + args.steps - 1} of the seeded trajectory, {len(probes)} probes, "
                f"{time.time() - t0:.0f} s"),
    }
    with open(OUT, "w") as f:
        json.dump(points, f, indent=1, sort_keys=True)
        f.write("\n")
    print(json.dumps(points[wl.name]))


if __name__ == "__main__":
    main()
