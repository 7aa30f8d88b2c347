#!/usr/bin/env python3
"""Benchmark of the GB300 branch-cached MoE layer stack (MoECa).

A step is one denoising step of the whole stack (every layer: router, select,
compact, grouped FFN, combine) over one batch of synthetic tokens.  The
headline workload is the 12-layer stack D 768, E 16, top-2, F 3072, T 2048
(8 x 256 tokens) in bf16, driven along its seeded drift trajectory, at the
60% branch-reuse point: tau0 calibrated on the oracle (oracle/calibrate_tau0.py,
stored in paper_2606_15615_gb300/headline_points.json) so that this GPU arm
and the reference arm (the oracle) time the same configuration.  The line
carries the sweep over reuse 0/30/60/90%, end-to-end numbers through the
host-buffer C call, a roofline entry for the dominant kernel, the oracle's CPU
baseline, the SM clocks sampled during the timed region, and one row per
other workload (the fp32 layer, the 28-layer and 16-layer stacks at 60%
reuse, the 64-expert layer over reuse 0-95% in 5% steps).

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]

Under torchrun every rank runs its own replica (the path shares nothing
between GPUs); the time is the max over ranks and the value sums the tokens.
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
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

METRIC = "branch-cached MoE layer tokens/s and effective TFLOP/s vs reuse ratio; % roofline"
DEFAULT_WORKLOAD = "moe_d768_e16_k2_f3072_t2048_l12_bf16"
FALLBACK_PEAKS = {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0}
KINDS = ["router", "select", "compact", "ffn1", "ffn2", "combine", "prep", "ffn", "qkv", "attn", "oproj", "attn_aux",
         "adaln"]
# Reuse points per workload index (the measured reuse sweep of each workload) and the point each
# row's kernels are timed at.
CONFIG_POINTS = {1: (0.5,), 2: (0.0, 0.3, 0.6, 0.9), 3: (0.6,), 4: (0.6,),
                 5: tuple(round(0.05 * j, 2) for j in range(20))}
MAIN_POINT = {1: 0.5, 2: 0.6, 3: 0.6, 4: 0.6, 5: 0.6}
HEADLINE_POINTS = os.path.join(ROOT, "paper_2606_15615_gb300", "headline_points.json")


def headline_point(wl, reuse: float):
    """The stored oracle-calibrated tau0 of ``wl`` at ``reuse``, or None."""
    if not os.path.exists(HEADLINE_POINTS):
        return None
    with open(HEADLINE_POINTS) as f:
        pts = json.load(f)
    p = pts.get(wl.name)
    if p and abs(p.get("reuse_target", -1) - reuse) < 1e-9:
        return p
    return None


# ---------------------------------------------------------------------------
# ranks
# ---------------------------------------------------------------------------

def dist_env():
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return world, rank, local


def init_group(world: int, backend: str):
    if world <= 1:
        return None
    import torch.distributed as dist
    if not dist.is_initialized():
        dist.init_process_group(backend=backend)
    return dist


def aggregate(elapsed_ms: float, tokens: int, dist, device=None):
    """Max time and summed tokens over ranks (barrier-bracketed timing)."""
    if dist is None:
        return elapsed_ms, tokens
    import torch
    t = torch.tensor([elapsed_ms], dtype=torch.float64, device=device)
    n = torch.tensor([float(tokens)], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    dist.all_reduce(n, op=dist.ReduceOp.SUM)
    return float(t.item()), int(n.item())


# ---------------------------------------------------------------------------
# clocks during the timed region
# ---------------------------------------------------------------------------

class ClockSampler:
    QUERY = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
             "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
             "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_id: str):
        self.gpu_id = gpu_id
        self.proc = None
        self.path = None

    def start(self):
        import tempfile
        fd, self.path = tempfile.mkstemp(prefix="moeca_clocks_", suffix=".csv")
        os.close(fd)
        try:
            self.f = open(self.path, "w")
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--query-gpu={self.QUERY}", "--format=csv,noheader,nounits", "-lms", "100",
                 "-i", self.gpu_id], stdout=self.f, stderr=subprocess.DEVNULL)
        except OSError:
            self.proc = None
        time.sleep(0.3)

    def stop(self) -> dict:
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        time.sleep(0.25)
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        self.f.close()
        rows = []
        with open(self.path) as f:
            for line in f:
                parts = [p.strip() for p in line.split(",")]
                if len(parts) >= 9:
                    rows.append(parts)
        os.unlink(self.path)
        if not rows:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["no samples"]}

        def num(v):
            try:
                return float(v)
            except ValueError:
                return None
        sm = [num(r[1]) for r in rows if num(r[1])]
        mx = [num(r[2]) for r in rows if num(r[2])]
        pw = [num(r[3]) for r in rows if num(r[3])]
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[j] for r in rows for j in range(4) if r[5 + j].lower() == "active"})
        load = [s for s, p in zip(sm, pw) if pw and p > 0.5 * max(pw)] or sm
        return {"sm_mhz": statistics.median(load) if load else None, "sm_max_mhz": max(mx) if mx else None,
                "reasons": reasons, "samples": len(rows), "power_w_max": max(pw) if pw else None}


def gpu_smi_id(dev_index: int) -> str:
    import torch
    try:
        u = str(torch.cuda.get_device_properties(dev_index).uuid)
        return u if u.startswith("GPU-") else "GPU-" + u
    except Exception:
        return str(dev_index)


# ---------------------------------------------------------------------------
# peaks, traffic
# ---------------------------------------------------------------------------

def peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        with open(p) as f:
            d = json.load(f)
        return d, "measured"
    return dict(FALLBACK_PEAKS), "fallback"


def kernel_source_sha(kind: str) -> str:
    """First 16 hex digits of sha256 over the kernel's .cu file and the local
    headers it includes (so a recorded ncu figure expires with the code)."""
    fname = {"ffn1": "ffn_tc.cu", "ffn2": "ffn_tc.cu", "ffn": "ffn_tc.cu", "router": "router.cu", "select": "select.cu",
             "compact": "select.cu", "combine": "combine.cu", "prep": "prep.cu", "qkv": "proj_tc.cu",
             "oproj": "proj_tc.cu", "attn": "attention.cu", "attn_aux": "attention.cu", "adaln": "adaln.cu"}[kind]
    csrc = os.path.join(ROOT, "paper_2606_15615_gb300", "csrc")
    h = hashlib.sha256()
    with open(os.path.join(csrc, fname), "rb") as f:
        src = f.read()
    h.update(src)
    for inc in sorted(set(re.findall(rb'#include "([^"]+\.cuh)"', src))):
        with open(os.path.join(csrc, inc.decode()), "rb") as f:
            h.update(f.read())
    return h.hexdigest()[:16]


def recorded_traffic(kind: str, workload: str, reuse_target: float):
    """DRAM bytes per launch from a committed ncu summary, if the kernel is unchanged."""
    p = os.path.join(ROOT, "profiles", "traffic.json")
    if not os.path.exists(p):
        return None
    with open(p) as f:
        d = json.load(f)
    for e in d.get("entries", []):
        if (e.get("kernel") == kind and e.get("workload") == workload
                and abs(e.get("reuse_target", -1) - reuse_target) < 1e-6
                and e.get("source_sha") == kernel_source_sha(kind)):
            return e.get("dram_bytes_per_launch")
    return None


# ---------------------------------------------------------------------------
# the GPU runner
# ---------------------------------------------------------------------------

class Runner:
    """One workload on one GPU.  With ``shard = (rank, world)`` the handle
    holds this rank's contiguous slice of the batch and every step is a
    token-sharded step whose per-layer exchange is an NCCL all-gather."""

    def __init__(self, wl, device_index: int, n_steps: int, tile_n: int = 0, split_k: int = 0, shard=None,
                 combine_staged: bool = False, prefetch_mb=None):
        import numpy as np
        import torch
        from paper_2606_15615_gb300 import build
        build.build()
        from paper_2606_15615_gb300 import moeca as M
        from paper_2606_15615_gb300 import workloads as W
        self.torch, self.M, self.W, self.np = torch, M, W, np
        self.wl = wl
        self.shard = shard
        self.n_local = wl.n_tokens // shard[1] if shard else wl.n_tokens
        self.dev = torch.device("cuda", device_index)
        torch.cuda.set_device(self.dev)
        self.weights = [W.make_layer_weights_device(wl, l, self.dev) for l in range(wl.n_layers)]
        cfg = M.moeca_config_default(
            n_layers=wl.n_layers, hidden=wl.hidden, ffn=wl.ffn, n_experts=wl.n_experts, top_k=wl.top_k,
            n_shared=wl.n_shared, max_tokens=self.n_local,
            dtype=M.MOECA_BF16 if wl.dtype == "bf16" else M.MOECA_F32, refresh_period=wl.refresh_period,
            ffn_tile_n=tile_n, ffn_split_k=split_k, n_heads=wl.n_heads, seq_len=wl.seq if wl.n_heads else 0,
            adaln=int(wl.adaln), combine_direct=0 if combine_staged else 1)
        if prefetch_mb is not None:
            cfg.weight_prefetch_mb = prefetch_mb
        self.cfg = cfg
        self.stack = M.Stack(cfg, self.weights, device=device_index)
        dt = torch.bfloat16 if wl.dtype == "bf16" else torch.float32
        self.dt = dt
        xs = [torch.from_numpy(x) for x in W.trajectory(wl, n_steps)]
        if shard:  # this rank's rows of every step's batch
            xs = [x[shard[0] * self.n_local:(shard[0] + 1) * self.n_local] for x in xs]
            self.exchange = M.torch_allgather()
        self.x_host = torch.stack(xs).to(dt).pin_memory()
        self.x_dev = self.x_host.to(self.dev)
        T, D = self.n_local, wl.hidden
        self.out = torch.empty((T, D), dtype=dt, device=self.dev)
        self.stream = torch.cuda.current_stream(self.dev)
        # End to end through moeca_step_host: pinned host outputs, two of them
        # so that a step's read-back never waits for the one before.
        self.out_host = [torch.empty((T, D), dtype=dt).pin_memory() for _ in range(2)]
        # AdaLN workloads: a conditioning vector per sample and step, and the
        # Eq. 1 update of each step's output (x_t kept in float32; the noise
        # draw z is one fixed buffer, an input of the update).
        self.cond_host = self.cond_dev = None
        if wl.adaln:
            c = torch.from_numpy(W.workload_conditioning(wl, n_steps))
            self.cond_host = c.pin_memory()
            self.cond_dev = c.to(self.dev)
            g = torch.Generator(device=self.dev)
            g.manual_seed(3000 + wl.index)
            self.x_state = torch.empty((T, D), dtype=torch.float32, device=self.dev).normal_(generator=g)
            self.z = torch.empty((T, D), dtype=torch.float32, device=self.dev).normal_(generator=g)
            _, self.alpha, self.abar, self.beta = M.moeca_ddpm_schedule(max(wl.n_steps, n_steps, 2))

    def close(self):
        self.stack.close()
        self.weights = self.x_dev = self.x_host = self.out = self.out_host = None
        self.cond_dev = self.cond_host = None
        self.torch.cuda.synchronize(self.dev)
        self.torch.cuda.empty_cache()

    def _sampler_update(self, t, eps):
        """Eq. 1: x_{t-1} from x_t and this step's output; run step t visits schedule step n - 1 - t."""
        j = len(self.alpha) - 1 - (t % len(self.alpha))
        sigma = math.sqrt(self.beta[j]) if j > 0 else 0.0
        self.M.ddpm_step(self.x_state, eps, self.alpha[j], self.abar[j], sigma, z=self.z if sigma else None,
                         x_prev=self.x_state, stream=self.stream.cuda_stream)

    def _step(self, h, x_ptr, out, t, tau0, sp, cond=None):
        if self.shard:
            x = self.x_dev[t] if x_ptr == self.x_dev[t].data_ptr() else None
            assert x is not None, "token-sharded steps read the device trajectory"
            self.stack.step_sharded(x, t, self.shard[0], self.shard[1], self.exchange, tau0=tau0, out=out)
            return
        cp = None
        if self.wl.adaln:
            cp = (self.cond_dev[t] if cond is None else cond).data_ptr()
        self.M.moeca_step(h, x_ptr, out.data_ptr(), self.n_local, t, False, tau0, sp, cp)
        if self.wl.adaln:
            self._sampler_update(t, out)

    def _run(self, tau0, W_, K, kernel_timing=False, e2e=False):
        torch, M = self.torch, self.M
        h = self.stack.handle
        M.moeca_reset(h)
        M.moeca_set_kernel_timing(h, False)
        sp = self.stream.cuda_stream
        for t in range(W_):
            self._step(h, self.x_dev[t].data_ptr(), self.out, t, tau0, sp)
        torch.cuda.synchronize(self.dev)
        M.moeca_reset_stats(h)
        if kernel_timing:
            M.moeca_get_kernel_times(h, reset=True)
            M.moeca_set_kernel_timing(h, True)
        e0 = torch.cuda.Event(enable_timing=True)
        e1 = torch.cuda.Event(enable_timing=True)
        e0.record(self.stream)
        if e2e:
            self._e2e_steps(tau0, W_, K)
        else:
            for t in range(W_, W_ + K):
                self._step(h, self.x_dev[t].data_ptr(), self.out, t, tau0, sp)
        e1.record(self.stream)
        torch.cuda.synchronize(self.dev)
        ms = e0.elapsed_time(e1)
        kt = None
        if kernel_timing:
            M.moeca_set_kernel_timing(h, False)
            kt = M.moeca_get_kernel_times(h, reset=True)
        st = M.moeca_get_stats(h)
        return ms, st, kt

    def _e2e_steps(self, tau0, W_, K):
        """Steps W_ .. W_ + K - 1 through the host-buffer C call: each step's
        input is uploaded from pinned host memory and its output read back
        into pinned host memory by the library (moeca_step_host), which
        overlaps them with the neighbouring steps' compute; the join orders
        the end event after the last read-back."""
        M, h, sp = self.M, self.stack.handle, self.stream.cuda_stream
        if self.wl.adaln:
            return self._e2e_steps_sampler(tau0, W_, K)
        for t in range(W_, W_ + K):
            M.moeca_step_host(h, self.x_host[t].data_ptr(), self.out_host[t % 2].data_ptr(), self.wl.n_tokens, t,
                              False, tau0, sp)
        M.moeca_host_join(h, sp)

    def _e2e_steps_sampler(self, tau0, W_, K):
        """AdaLN workloads, whose step ends with the Eq. 1 update of the
        device output: the inputs and conditioning are uploaded and the
        outputs read back by torch copies on a side stream, double-buffered
        against the neighbouring steps (step t reads in_bufs[t % 2])."""
        torch = self.torch
        h, T, D, sp = self.stack.handle, self.wl.n_tokens, self.wl.hidden, self.stream.cuda_stream
        in_bufs = [torch.empty((T, D), dtype=self.dt, device=self.dev) for _ in range(2)]
        out_bufs = [torch.empty((T, D), dtype=self.dt, device=self.dev) for _ in range(2)]
        cond_bufs = [torch.empty_like(self.cond_dev[0]) for _ in range(2)]
        cs = torch.cuda.Stream(device=self.dev)
        ev = lambda: torch.cuda.Event()  # noqa: E731
        up, done, back = [ev(), ev()], [ev(), ev()], [ev(), ev()]
        cs.wait_stream(self.stream)
        with torch.cuda.stream(cs):
            in_bufs[W_ % 2].copy_(self.x_host[W_], non_blocking=True)
            cond_bufs[W_ % 2].copy_(self.cond_host[W_], non_blocking=True)
            up[W_ % 2].record(cs)
        for t in range(W_, W_ + K):
            b = t % 2
            self.stream.wait_event(up[b])
            if t - 2 >= W_:
                self.stream.wait_event(back[b])
            self._step(h, in_bufs[b].data_ptr(), out_bufs[b], t, tau0, sp, cond=cond_bufs[b])
            done[b].record(self.stream)
            with torch.cuda.stream(cs):
                if t + 1 < W_ + K:
                    nb = (t + 1) % 2
                    if t - 1 >= W_:
                        cs.wait_event(done[nb])
                    in_bufs[nb].copy_(self.x_host[t + 1], non_blocking=True)
                    cond_bufs[nb].copy_(self.cond_host[t + 1], non_blocking=True)
                    up[nb].record(cs)
                cs.wait_event(done[b])
                self.out_host[b].copy_(out_bufs[b], non_blocking=True)
                back[b].record(cs)
        self.stream.wait_stream(cs)

    def reuse_of(self, st) -> float:
        return st["reused"] / max(st["branches"], 1)

    def calibrate(self, target: float, W_, K) -> tuple:
        """tau0 whose reuse over the timed window is closest to ``target`` (bisection)."""
        if target <= 0.0:
            _, st, _ = self._run(-math.inf, W_, K)
            return -math.inf, self.reuse_of(st)
        lo, hi = 0.0, 4.0
        _, st_hi, _ = self._run(hi, W_, K)
        if self.reuse_of(st_hi) <= target:
            return hi, self.reuse_of(st_hi)
        best = (hi, self.reuse_of(st_hi))
        for _ in range(14):
            mid = 0.5 * (lo + hi)
            _, st, _ = self._run(mid, W_, K)
            r = self.reuse_of(st)
            if abs(r - target) < abs(best[1] - target):
                best = (mid, r)
            if r < target:
                lo = mid
            else:
                hi = mid
        return best


def algorithmic(kind: str, wl, rows_per_launch: float, active_groups: float, attn_rows: float = 0.0):
    """Algorithmic (bytes, flops) of one launch of a kernel kind for this workload.

    ``rows_per_launch`` is the mean number of recomputed branch rows (plus
    shared-expert rows) of one layer step; ``attn_rows`` the mean number of
    token rows one attention launch computes (every token on a full step, the
    recomputing tokens otherwise).  The FFN's bf16 hidden activations are
    an implementation intermediate, not algorithmic: its bytes are the active
    experts' weights, the gathered input rows and the scattered output rows."""
    T, D, E, k, F, S = wl.n_tokens, wl.hidden, wl.n_experts, wl.top_k, wl.ffn, wl.n_shared
    es = 2 if wl.dtype == "bf16" else 4
    if kind == "qkv":      # x [T, D] and W_qkv [3D, D] in, q | k | v [T, 3D] out
        return T * D * es + 3 * D * D * es + 3 * D * 4 + 3 * T * D * es, 2.0 * T * D * 3 * D
    if kind == "attn":     # q rows, every key and value row once, o rows
        return 2 * attn_rows * D * es + 2 * T * D * es, 4.0 * attn_rows * wl.seq * D
    if kind == "oproj":    # o rows and W_o in; x rows in; a and u rows out
        return 4 * attn_rows * D * es + D * D * es + D * 4, 2.0 * attn_rows * D * D
    if kind == "attn_aux":  # u = x + a^{t0} (x, a in, u out), the token list, the FFN row gather
        return 3 * T * D * es + T + rows_per_launch * 2 * D * es, 0.0
    if kind == "adaln":
        # Mean over a cache step's 1 + 2L launches: the modulation GEMV (every
        # layer's W_ada once), then per layer the row pass (x, a^{t0} in; u',
        # m', h out) and the recomputing rows' m = LN-modulate(u).
        L, B = wl.n_layers, wl.batch
        mod = L * 6 * D * D * es + L * 6 * D * 4 + B * D * 4 + L * B * 6 * D * 4
        pre = 5 * T * D * es + B * 6 * D * 4
        mrows = attn_rows * (2 * D * es + 4)
        return (mod + L * (pre + mrows)) / (1 + 2 * L), 2.0 * L * B * 6 * D * D / (1 + 2 * L)
    if kind == "router":
        return T * D * es + E * D * es + T * E * 8 + T * k * 8, 2.0 * T * D * E
    if kind == "select":
        return T * k * (8 + 12 + 8 + 3) + T, 0.0
    if kind == "compact":
        return T * k * 6 + T + rows_per_launch * (4 + 2 * D * es), 0.0
    if kind == "ffn1":     # W1 of the active experts, gathered input rows
        return active_groups * F * D * es + rows_per_launch * D * es, 2.0 * rows_per_launch * D * F
    if kind == "ffn2":     # W2 of the active experts, output rows scattered into the cache
        return active_groups * F * D * es + rows_per_launch * D * es, 2.0 * rows_per_launch * D * F
    if kind == "ffn":
        b1, f1 = algorithmic("ffn1", wl, rows_per_launch, active_groups)
        b2, f2 = algorithmic("ffn2", wl, rows_per_launch, active_groups)
        return b1 + b2, f1 + f2
    if kind == "combine":
        return T * D * es * (2 + k + S) + T * k * 9, 0.0
    if kind == "prep":
        return (algorithmic("router", wl, rows_per_launch, active_groups)[0]
                + algorithmic("select", wl, rows_per_launch, active_groups)[0]
                + algorithmic("compact", wl, rows_per_launch, active_groups)[0],
                algorithmic("router", wl, rows_per_launch, active_groups)[1])
    raise KeyError(kind)


def kernel_table(wl, kt, st_k, K):
    """Per-kernel-kind mean event time, algorithmic bytes / flops and achieved rates."""
    rows_per_launch = (st_k["recomputed"] + st_k["shared_recomputed"]) / (K * wl.n_layers)
    attn_rows = st_k["attn_recomputed"] / max(kt["attn"][1], 1)
    total = max(sum(v[0] for v in kt.values()), 1e-12)
    kernels = {}
    for kind in KINDS:
        tot, n = kt[kind]
        if not n:
            continue
        nb, nf = algorithmic(kind, wl, rows_per_launch, wl.n_experts + wl.n_shared, attn_rows)
        avg = tot / n
        kernels[kind] = {"launches": n, "avg_us": avg * 1e3, "share": tot / total, "alg_bytes": nb, "alg_flops": nf,
                         "gbs": nb / (avg * 1e-3) / 1e9 if avg > 0 else None,
                         "tflops": nf / (avg * 1e-3) / 1e12 if avg > 0 and nf else None}
    return kernels


def roofline(kind: str, kd: dict, wl, pk: dict, pk_src: str, ffma_peak):
    """Roofline entry of one kernel kind from its event-timed mean.

    Peaks are MEASURED_PEAKS.json's burst figures (the kernels are timed one
    launch at a time): HBM copy GB/s and cuBLAS bf16 TFLOP/s.  A bf16 kernel
    whose algorithmic intensity is above the ridge is tensor-bound; the fp32
    path's FFN is FFMA-bound, against the measured FFMA rate.  Both fractions
    are given for the FFN."""
    src = "of measured (MEASURED_PEAKS.json, burst)" if pk_src == "measured" else "of fallback"
    ridge = pk["bf16_tflops"] * 1e12 / (pk["hbm_gbs"] * 1e9)
    hbm = {"achieved": kd["gbs"], "peak": pk["hbm_gbs"], "unit": "GB/s",
           "frac": kd["gbs"] / pk["hbm_gbs"] if kd["gbs"] else None}
    r = {"kernel": kind, "alg_bytes_per_launch": kd["alg_bytes"], "alg_flops_per_launch": kd["alg_flops"],
         "avg_us": kd["avg_us"]}
    if wl.dtype != "bf16" and kind in ("ffn1", "ffn2") and ffma_peak:
        tf = kd["tflops"]
        r.update(bound="fp32", achieved=tf, peak=ffma_peak, unit="TFLOP/s", frac=tf / ffma_peak if tf else None,
                 peak_source="measured on this GPU (moeca_probe_ffma)", hbm=hbm)
    elif kd["alg_flops"] and kd["alg_flops"] / kd["alg_bytes"] > ridge:
        tf = kd["tflops"]
        r.update(bound="tensor", achieved=tf, peak=pk["bf16_tflops"], unit="TFLOP/s",
                 frac=tf / pk["bf16_tflops"] if tf else None, peak_source=src, hbm=hbm)
    else:
        r.update(bound="hbm", achieved=hbm["achieved"], peak=hbm["peak"], unit="GB/s", frac=hbm["frac"],
                 peak_source=src)
        if kd["alg_flops"] and kd["tflops"]:
            r["tensor"] = {"achieved": kd["tflops"], "peak": pk["bf16_tflops"], "unit": "TFLOP/s",
                           "frac": kd["tflops"] / pk["bf16_tflops"]}
    return r


def stream_ceiling(M, wl, device: int, kd, pk: dict) -> dict:
    """What a plain streaming kernel reaches at the combine's size and shape
    (moeca_probe_stream: a token's k + shared + 1 rows read, one written, one
    warp per token, clean L2), beside the combine's event-timed rate: at tens
    of MB a launch's ramp and drain keep any kernel below the large-copy peak."""
    es = 2 if wl.dtype == "bf16" else 4
    rows = wl.top_k + wl.n_shared + 1
    gbs, us = M.moeca_probe_stream(device, wl.n_tokens, rows, wl.hidden * es)
    return {"shape": f"{wl.n_tokens} tokens x {rows} rows of {wl.hidden * es} B read, one row written",
            "stream_gbs": gbs, "stream_us": us, "stream_frac_of_peak": gbs / pk["hbm_gbs"],
            "combine_gbs": kd["gbs"], "combine_frac_of_stream": kd["gbs"] / gbs if kd["gbs"] else None}


def point_row(runner, wl, tgt, tau0, ms, st, K, world):
    tokens_all = wl.n_tokens * K * world
    executed = (st["recomputed"] + st["shared_recomputed"]) * 4.0 * wl.hidden * wl.ffn
    dense = wl.dense_flops_per_layer() * wl.n_layers * K
    if wl.n_heads:
        D, T = wl.hidden, wl.n_tokens
        executed += (2.0 * T * D * 3 * D * wl.n_layers * K
                     + st["attn_recomputed"] * (4.0 * wl.seq * D + 2.0 * D * D))
        dense += (2.0 * T * D * 3 * D + T * (4.0 * wl.seq * D + 2.0 * D * D)) * wl.n_layers * K
    return {"reuse_target": tgt, "reuse_achieved": round(runner.reuse_of(st), 4),
            "tau0": None if not math.isfinite(tau0) else round(tau0, 5), "tokens_per_s": tokens_all / (ms / 1e3),
            "ms_per_step": ms / K, "effective_tflops": dense * world / (ms / 1e3) / 1e12,
            "executed_tflops": executed * world / (ms / 1e3) / 1e12}


def config_row(wl, local: int, W_: int, K: int, pk, pk_src, ffma_peak):
    """One benchmark workload at its reuse points: tokens/s, effective TFLOP/s
    per point, and at the main point the per-kernel times with the dominant
    kernel's roofline."""
    runner = Runner(wl, local, W_ + K)
    try:
        pts, main = CONFIG_POINTS[wl.index], MAIN_POINT[wl.index]
        rows, main_tau = [], None
        for tgt in pts:
            tau0, _ = runner.calibrate(tgt, W_, K)
            reps = [runner._run(tau0, W_, K) for _ in range(2)]
            ms = statistics.median(r[0] for r in reps)
            rows.append(point_row(runner, wl, tgt, tau0, ms, reps[-1][1], K, 1))
            if abs(tgt - main) < 1e-9:
                main_tau = tau0
        _, st_k, kt = runner._run(main_tau, W_, K, kernel_timing=True)
        kernels = kernel_table(wl, kt, st_k, K)
        dom = max(kernels, key=lambda k_: kernels[k_]["avg_us"] * kernels[k_]["launches"])
        row = {"workload": wl.name, "dtype": wl.dtype, "tokens": wl.n_tokens, "layers": wl.n_layers,
               **next(r for r in rows if abs(r["reuse_target"] - main) < 1e-9),
               "roofline": roofline(dom, kernels[dom], wl, pk, pk_src, ffma_peak),
               "kernels": {k_: {kk: (round(v, 3) if isinstance(v, float) else v) for kk, v in d.items()
                                if kk in ("launches", "avg_us", "share", "gbs", "tflops")}
                           for k_, d in kernels.items()}}
        for kind in ("ffn", "ffn2", "combine", "prep", "router"):
            if kind in kernels and kind != dom:
                row[f"roofline_{kind}"] = roofline(kind, kernels[kind], wl, pk, pk_src, ffma_peak)
        if "combine" in kernels:
            row["combine_size_ceiling"] = stream_ceiling(runner.M, wl, local, kernels["combine"], pk)
        if len(rows) > 1:
            row["sweep"] = rows
        return row
    finally:
        runner.close()


def cpu_oracle_baseline(wl, runner, tau0: float, budget_s: float = 12.0):
    """The oracle on this host's cores: full-T cache steps of layer 0, extrapolated to L layers."""
    import numpy as np
    from oracle import moeca_oracle as O
    w = {k: (None if v is None else v.float().cpu().numpy().astype(np.float64)) for k, v in runner.weights[0].items()}
    if w["ws1"] is None:
        w["ws1"] = w["ws2"] = None
    prm = O.Params(top_k=wl.top_k, tau0=tau0 if math.isfinite(tau0) else tau0, refresh_period=wl.refresh_period,
                   n_heads=wl.n_heads, seq_len=wl.seq if wl.n_heads else 0, adaln=wl.adaln,
                   act_store="bf16" if wl.adaln else "f64")
    st = O.Stack([w], prm, wl.hidden, wl.n_experts, wl.n_shared)
    xs = runner.x_host.float().numpy()
    conds = runner.cond_host.numpy().astype(np.float64) if wl.adaln else [None] * xs.shape[0]
    st.step(xs[0], 0, cond=conds[0])
    times = []
    t_all = time.perf_counter()
    for t in range(1, xs.shape[0]):
        if wl.refresh_period and t % wl.refresh_period == 0:
            st.step(xs[t], t, cond=conds[t])
            continue
        t0 = time.perf_counter()
        st.step(xs[t], t, cond=conds[t])
        times.append(time.perf_counter() - t0)
        if time.perf_counter() - t_all > budget_s:
            break
    per_layer = statistics.mean(times)
    return {"value": wl.n_tokens / (per_layer * wl.n_layers), "unit": "tokens/s", "cores": host_threads(),
            "kind": "oracle",
            "sample": (f"{len(times)} cache steps of layer 0 at full T={wl.n_tokens} (tau0 of the headline point), "
                       f"{per_layer * 1e3:.0f} ms per layer step, extrapolated to {wl.n_layers} layers; "
                       f"numpy float64, host cores {os.cpu_count()}")}


def host_threads() -> int:
    try:
        from threadpoolctl import threadpool_info
        return max([i.get("num_threads", 1) for i in threadpool_info()] or [1])
    except Exception:
        return os.cpu_count()


# ---------------------------------------------------------------------------
# the reference arm: the oracle on host cores
# ---------------------------------------------------------------------------

def reference_arm(args, wl):
    """The oracle (plain numpy float64) on the host cores: the whole L-layer
    stack on consecutive steps of the same seeded trajectory, with the same
    weights (torch's seeded CUDA generator, copied to host memory) and the
    same headline tau0 as the GPU arm; W untimed steps, then K timed ones."""
    import numpy as np
    import torch
    from oracle import moeca_oracle as O
    from paper_2606_15615_gb300 import workloads as W
    pt = headline_point(wl, args.reuse)
    tau0 = args.tau0 if args.tau0 is not None else (pt["tau0"] if pt else args.ref_tau0)
    dev = torch.device("cuda", 0) if torch.cuda.is_available() else None
    ws = []
    for l in range(wl.n_layers):
        if dev is not None:
            w = W.make_layer_weights_device(wl, l, dev)
            w = {k: (None if v is None else v.float().cpu().numpy().astype(np.float64)) for k, v in w.items()}
        else:
            w = W.make_layer_weights(wl, l)
        if wl.n_heads:
            w.update(W.make_attn_weights(wl, l))
            if wl.adaln:
                w.update(W.make_adaln_weights(wl, l))
        ws.append(w)
    xs = list(W.trajectory(wl, args.warmup + args.steps))
    conds = W.workload_conditioning(wl, len(xs)) if wl.adaln else [None] * len(xs)
    prm = O.Params(top_k=wl.top_k, tau0=tau0, refresh_period=wl.refresh_period,
                   n_heads=wl.n_heads, seq_len=wl.seq if wl.n_heads else 0, adaln=wl.adaln,
                   act_store="bf16" if wl.adaln else "f64")
    stack = O.Stack(ws, prm, wl.hidden, wl.n_experts, wl.n_shared)
    for t in range(args.warmup):
        stack.step(xs[t], t, cond=conds[t])
    reused = routed = 0
    t0 = time.perf_counter()
    for t in range(args.warmup, args.warmup + args.steps):
        _, infos = stack.step(xs[t], t, cond=conds[t])
        for inf in infos:
            reused += int((~inf["recompute"]).sum())
            routed += inf["recompute"].size
    elapsed = time.perf_counter() - t0
    value = wl.n_tokens * args.steps / elapsed
    cores = host_threads()
    line = {
        "impl": "reference", "metric": METRIC, "value": value, "unit": "tokens/s", "n_gpus": args.gpus,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": elapsed / args.steps * 1e3,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "config": {"workload": wl.name, "reuse_target": args.reuse},
        "point": {"tau0": tau0, "tau0_source": "oracle-calibrated (headline_points.json)" if pt and args.tau0 is None
                  else "command line", "reuse_achieved": round(reused / max(routed, 1), 4)},
        "cpu_baseline": {"value": value, "unit": "tokens/s", "cores": cores, "kind": "oracle",
                         "sample": (f"the whole {wl.n_layers}-layer stack, {args.steps} consecutive timed steps "
                                    f"after {args.warmup} untimed ones, at full T={wl.n_tokens}; numpy float64 on "
                                    f"{os.cpu_count()} host cores; no extrapolation")},
        "e2e": {"value": value, "unit": "tokens/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line))


# ---------------------------------------------------------------------------
# token-sharded stacks across ranks
# ---------------------------------------------------------------------------

def sharded_main(args, wl, world, rank, local, dist):
    """The workload's batch split by tokens over the ranks: every step runs
    the token-sharded step, each layer exchanging its entropy partials with an
    NCCL all-gather; the time is the max over ranks of K steps of the one
    batch (strong scaling: the work is fixed as N grows)."""
    import torch
    if wl.n_tokens % (32 * world):
        raise SystemExit(f"{wl.n_tokens} tokens do not split into {world} slices of whole 32-token blocks")
    runner = Runner(wl, local, args.warmup + args.steps, args.ffn_tile_n, args.ffn_split_k, shard=(rank, world),
                    combine_staged=args.combine_staged, prefetch_mb=args.weight_prefetch_mb)
    pt = headline_point(wl, args.reuse)
    tau0 = args.tau0 if args.tau0 is not None else (pt["tau0"] if pt else args.ref_tau0)
    W_, K = args.warmup, args.steps
    reps = []
    st = None
    for _ in range(args.reps):
        dist.barrier()
        torch.cuda.synchronize(runner.dev)
        ms, st, _ = runner._run(tau0, W_, K)
        ms, _ = aggregate(ms, 0, dist, runner.dev)
        reps.append(ms)
    ms = statistics.median(reps)
    n = torch.tensor([float(st["reused"]), float(st["branches"])], dtype=torch.float64, device=runner.dev)
    dist.all_reduce(n)
    line = {
        "metric": METRIC, "value": wl.n_tokens * K / (ms / 1e3), "unit": "tokens/s", "n_gpus": world, "steps": K,
        "warmup": W_, "ms_per_step": ms / K, "higher_is_better": True, "scaling": "strong", "vs_baseline": None,
        "dtype": wl.dtype, "data": "synthetic",
        "config": {"workload": wl.name, "reuse_target": args.reuse, "parallelism": f"token-sharded x{world}"},
        "point": {"tau0": tau0, "reuse_achieved": round(float(n[0] / max(n[1], 1)), 4)},
        "exchange": f"one NCCL all-gather per layer per step of {world} x "
                    f"{runner.M.moeca_shard_exchange_bytes(runner.stack.handle, runner.n_local)} bytes "
                    "(per-block entropy partials)",
    }
    if rank == 0:
        print(json.dumps(line))
    dist.barrier()
    dist.destroy_process_group()
    runner.close()


# ---------------------------------------------------------------------------

def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=20)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--workload", default=DEFAULT_WORKLOAD)
    ap.add_argument("--reuse", type=float, default=0.6, help="headline reuse target")
    ap.add_argument("--no-sweep", action="store_true")
    ap.add_argument("--no-cpu", action="store_true", help="skip the CPU oracle baseline")
    ap.add_argument("--configs", default="auto",
                    help="other workloads to add as rows: 'all', 'none', or indices like '1,3' "
                         "(auto: all with the default workload, none otherwise)")
    ap.add_argument("--reps", type=int, default=5)
    ap.add_argument("--ref-tau0", type=float, default=0.665, help="reference arm tau0 without a stored point")
    ap.add_argument("--ffn-tile-n", type=int, default=0, help="force the tensor-core FFN tile width (0: auto)")
    ap.add_argument("--combine-staged", action="store_true",
                    help="stage the combine's rows in shared memory where they fit (default: the direct form)")
    ap.add_argument("--ffn-split-k", type=int, default=0, help="force the tensor-core FFN K splits (0: auto)")
    ap.add_argument("--weight-prefetch-mb", type=int, default=None,
                    help="MB of each layer's routed W1 the preparation kernel brings into L2 (default: the library's)")
    ap.add_argument("--tau0", type=float, default=None,
                    help="use this tau0 for the headline point instead of the stored / calibrated one")
    ap.add_argument("--layers", type=int, default=0,
                    help="run only the first N layers of the workload (small ncu captures; not a bench line)")
    ap.add_argument("--shard", action="store_true",
                    help="under torchrun: split each step's batch over the ranks by tokens (one NCCL all-gather of "
                         "the entropy partials per layer) instead of running one replica per rank")
    args = ap.parse_args()
    if args.warmup < 3:
        ap.error("--warmup must be >= 3")
    from paper_2606_15615_gb300 import workloads as W
    wl = W.workload(args.workload)
    if args.layers:
        wl = wl.scaled(n_layers=min(args.layers, wl.n_layers))
    world, rank, local = dist_env()

    if args.impl == "reference":
        if rank == 0:
            reference_arm(args, wl)
        return

    import torch
    dist = init_group(world, "nccl")
    if args.shard and world > 1:
        return sharded_main(args, wl, world, rank, local, dist)
    runner = Runner(wl, local, args.warmup + args.steps, args.ffn_tile_n, args.ffn_split_k,
                    combine_staged=args.combine_staged, prefetch_mb=args.weight_prefetch_mb)
    dev = runner.dev
    W_, K = args.warmup, args.steps
    targets = [args.reuse] if args.no_sweep else sorted(set(wl.reuse_targets) | {args.reuse})
    pk, pk_src = peaks()
    stored = headline_point(wl, args.reuse) if not args.layers else None
    sweep = []
    head = None
    for tgt in targets:
        is_head = abs(tgt - args.reuse) < 1e-9
        if is_head and args.tau0 is not None:
            tau0, src = args.tau0, "command line"
        elif is_head and stored is not None:
            tau0, src = stored["tau0"], "oracle-calibrated (headline_points.json)"
        else:
            tau0, _ = runner.calibrate(tgt, W_, K)
            src = "calibrated on this GPU"
        sampler = None
        if is_head and rank == 0:
            sampler = ClockSampler(gpu_smi_id(local))
            sampler.start()
        reps = []
        st = None
        for _ in range(args.reps if is_head else 2):
            if dist is not None:
                dist.barrier()
            torch.cuda.synchronize(dev)
            ms, st, _ = runner._run(tau0, W_, K)
            ms, _ = aggregate(ms, wl.n_tokens * K, dist, dev)
            reps.append(ms)
        clocks = sampler.stop() if sampler else None
        row = point_row(runner, wl, tgt, tau0, statistics.median(reps), st, K, world)
        sweep.append(row)
        if is_head:
            head = dict(row, clocks=clocks, stats=st, tau0_raw=tau0, tau0_source=src)

    # Per-kernel CUDA-event durations on the launching stream, same steps as the headline.
    _, st_k, kt = runner._run(head["tau0_raw"], W_, K, kernel_timing=True)
    # End to end through the host-buffer C call.
    if dist is not None:
        dist.barrier()
    e2e_reps = [runner._run(head["tau0_raw"], W_, K, e2e=True)[0] for _ in range(max(1, args.reps))]
    e2e_ms, _ = aggregate(statistics.median(e2e_reps), 0, dist, dev)
    kernels = kernel_table(wl, kt, st_k, K)
    ffma_peak = None
    if wl.dtype != "bf16" or args.configs != "none":
        ffma_peak = runner.M.moeca_probe_ffma(local)[0]
    dom = max(kernels, key=lambda k_: kernels[k_]["avg_us"] * kernels[k_]["launches"])
    roof = roofline(dom, kernels[dom], wl, pk, pk_src, ffma_peak)
    roof["traffic"] = recorded_traffic(dom, wl.name, args.reuse)
    ceiling = stream_ceiling(runner.M, wl, local, kernels["combine"], pk) if "combine" in kernels else None

    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu:
        cpu = cpu_oracle_baseline(wl, runner, head["tau0_raw"])
    es = 2 if wl.dtype == "bf16" else 4
    io_bytes = wl.n_tokens * wl.hidden * es
    cond_bytes = wl.batch * wl.hidden * 4 if wl.adaln else 0
    runner.close()

    # The other workloads, one row each (rank 0 of a single-GPU run).
    rows = []
    want = args.configs
    if want == "auto":
        want = "all" if (args.workload == DEFAULT_WORKLOAD and world == 1 and not args.layers) else "none"
    if want != "none" and rank == 0:
        idx = [1, 2, 3, 4, 5] if want == "all" else [int(v) for v in want.split(",") if v]
        for i in idx:
            if i == wl.index and not wl.n_heads:
                continue
            rows.append(config_row(W.workload(i), local, W_, K, pk, pk_src, ffma_peak))

    line = {
        "metric": METRIC, "value": head["tokens_per_s"], "unit": "tokens/s", "n_gpus": world, "steps": K,
        "warmup": W_, "ms_per_step": head["ms_per_step"], "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": wl.dtype, "data": "synthetic",
        "config": {"workload": wl.name, "reuse_target": args.reuse},
        "point": {"tau0": head["tau0"], "tau0_source": head["tau0_source"], "reuse_achieved": head["reuse_achieved"],
                  "effective_tflops": head["effective_tflops"], "executed_tflops": head["executed_tflops"]},
        "shape": {"tokens": wl.n_tokens, "hidden": wl.hidden, "experts": wl.n_experts,
                  "shared_experts": wl.n_shared, "top_k": wl.top_k, "ffn": wl.ffn, "layers": wl.n_layers,
                  "refresh_period": wl.refresh_period,
                  **({"attn_heads": wl.n_heads, "seq_len": wl.seq,
                      "attn_rows_recomputed_per_step": head["stats"]["attn_recomputed"] / K}
                     if wl.n_heads else {}),
                  **({"adaln": True,
                      "step": "AdaLN modulation of every block from the step's conditioning, the L blocks, "
                              "then the Eq. 1 update of the step's output (x_t in float32); the blocks' "
                              "inputs follow the synthetic drift trajectory, not the update, so the reuse "
                              "ratio is controlled as for the other workloads"}
                     if wl.adaln else {}),
                  "timed": f"median of {args.reps} reps of {K} steps after {W_} warm-up steps (step 0 full)",
                  "l2": "no flush: each step streams the active experts' weights "
                        f"({wl.n_layers} x {2 * wl.n_experts * wl.hidden * wl.ffn * es / 1e6:.0f} MB) > 129 MB L2",
                  "parallelism": f"replicas x{world}"},
        "roofline": roof,
        "combine_size_ceiling": ceiling,
        "cpu_baseline": cpu,
        "e2e": {"value": wl.n_tokens * K * world / (e2e_ms / 1e3), "unit": "tokens/s",
                "h2d_bytes_per_step": io_bytes + cond_bytes, "d2h_bytes_per_step": io_bytes,
                "how": ("torch copies on a side stream, double-buffered (the AdaLN step ends with the Eq. 1 "
                        "update of the device output)" if wl.adaln else
                        "moeca_step_host per step from pinned host input to pinned host output: the library "
                        "uploads on its own stream into double-buffered staging and reads back on another, so "
                        "the copies overlap the neighbouring steps' compute; moeca_host_join before the end event")},
        "gpu_launches": sum(kt[k_][1] for k_ in KINDS) + (K if wl.adaln else 0),
        "clocks": head["clocks"],
        "sweep": sweep,
        "kernels": kernels,
        "fp32_ffma_tflops": ffma_peak,
        "configs": rows,
    }
    if rank == 0:
        print(json.dumps(line))
    if dist is not None:
        dist.barrier()
        dist.destroy_process_group()


if __name__ == "__main__":
    main()
