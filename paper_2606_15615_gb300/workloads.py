"""Seeded synthetic workloads for the branch-cached DiT-MoE layer stack.

This module only makes inputs: layer shapes, Gaussian weights (rounded to bf16
where the workload is bf16), drift trajectories of the token activations that
enter the first layer, and a router bias that skews expert loads.  It holds none
of MoECa's arithmetic (no routing, scoring, thresholds or expert FFNs), so the
CUDA path and the CPU oracle can both draw their inputs from it without sharing
any of the method.

The shapes stand in for the paper's DiT-MoE models (DSMoE / DiT-MoE at 256px,
HiDream-I1 at 1024px, Sec. 5.1); the real checkpoints and datasets are not
used.  Every draw comes from numpy's PCG64 seeded with a tuple that names the
workload, the layer and the tensor, so any tensor can be regenerated alone.
"""
from __future__ import annotations

import math
from dataclasses import dataclass, replace

import numpy as np

# Seed roots: weights 1000 + workload index, trajectories 2000 + workload index.
_WEIGHT_SEED = 1000
_TRAJ_SEED = 2000

# Tensor ids inside a layer's weight seed tuple.
_T_GATE, _T_W1, _T_W2, _T_WS1, _T_WS2, _T_BIAS, _T_QKV, _T_BQKV, _T_WO, _T_BO, _T_ADA, _T_BADA = range(12)


@dataclass(frozen=True)
class Workload:
    """Shape and trajectory recipe of one synthetic MoE layer stack."""

    name: str
    index: int            # 1..5, selects the seed streams
    hidden: int           # D
    n_experts: int        # E (routed)
    top_k: int            # k
    ffn: int              # F, per routed expert (shared expert uses the same F)
    batch: int
    seq: int              # tokens per sample; T = batch * seq
    n_layers: int         # L
    n_steps: int          # denoising steps in the trajectory
    dtype: str            # "f32" or "bf16"
    n_shared: int = 0     # always-on shared experts (0 or 1)
    refresh_period: int = 0   # full-computation step every N steps (0: step 0 only)
    drift: str = "decay"      # "per_token" (sigma_i ~ U) or "decay" (sigma_t linear)
    router_skew: tuple = ()   # target top-k load shares, e.g. (4, 2, 1, 1)
    reuse_targets: tuple = (0.5,)
    n_heads: int = 0          # > 0: DiT-MoE blocks (self-attention over each sample's seq tokens, then MoE)
    adaln: bool = False       # DiT-MoE blocks with AdaLN modulation and a per-sample conditioning input

    @property
    def n_tokens(self) -> int:
        return self.batch * self.seq

    def scaled(self, **kw) -> "Workload":
        """Same recipe with some sizes replaced (small parity cases)."""
        return replace(self, **kw)

    def dense_flops_per_layer(self) -> float:
        """Flops of every routed and shared branch at 0% reuse (4*D*F per branch)."""
        return float(self.n_tokens * (self.top_k + self.n_shared) * 4 * self.hidden * self.ffn)


WORKLOADS = {
    # Single fp32 MoE-FFN layer, the debug-precision case.
    "moe_d384_e8_k2_f1536_t512_l1_f32": Workload(
        "moe_d384_e8_k2_f1536_t512_l1_f32", 1, 384, 8, 2, 1536, 2, 256, 1, 4, "f32",
        drift="per_token", reuse_targets=(0.5,)),
    # 12-layer stack at 256px (32x32 latent, patch 2), 8 images.
    "moe_d768_e16_k2_f3072_t2048_l12_bf16": Workload(
        "moe_d768_e16_k2_f3072_t2048_l12_bf16", 2, 768, 16, 2, 3072, 8, 256, 12, 50, "bf16",
        reuse_targets=(0.0, 0.3, 0.6, 0.9)),
    # 28-layer stack at 512px, full-computation step every 5 steps.
    "moe_d1152_e16_k2_f4608_t4096_l28_bf16": Workload(
        "moe_d1152_e16_k2_f4608_t4096_l28_bf16", 3, 1152, 16, 2, 4608, 4, 1024, 28, 50, "bf16",
        refresh_period=5, reuse_targets=(0.6,)),
    # 16-layer stack at 1024px with one shared expert and skewed routing.
    "moe_d2560_e4s1_k2_f6912_t4096_l16_bf16": Workload(
        "moe_d2560_e4s1_k2_f6912_t4096_l16_bf16", 4, 2560, 4, 2, 6912, 1, 4096, 16, 30, "bf16",
        n_shared=1, router_skew=(4, 2, 1, 1), reuse_targets=(0.6,)),
    # Fine-grained single layer: 64 experts, top-8, narrow experts.
    "moe_d1152_e64_k8_f768_t4096_l1_bf16": Workload(
        "moe_d1152_e64_k8_f768_t4096_l1_bf16", 5, 1152, 64, 8, 768, 4, 1024, 1, 20, "bf16",
        reuse_targets=tuple(round(0.05 * j, 2) for j in range(20))),
}

WORKLOAD_ORDER = list(WORKLOADS)

# Attention heads of the DiT models each bf16 stack stands in for: DiT-B (768,
# 12 x 64), DiT-XL (1152, 16 x 72), HiDream-I1 (2560, 20 x 128).
_HEADS = {384: 6, 768: 12, 1152: 16, 2560: 20}


def dit_variant(wl: Workload) -> Workload:
    """The same stack with every layer a DiT-MoE block (attention sub-layer first)."""
    name = wl.name.replace("moe_d%d_" % wl.hidden, "dit_d%d_h%d_" % (wl.hidden, _HEADS[wl.hidden]), 1)
    return replace(wl, name=name, n_heads=_HEADS[wl.hidden])


DIT_WORKLOADS = {d.name: d for d in (dit_variant(w) for w in WORKLOADS.values() if w.dtype == "bf16")}


def adaln_variant(wl: Workload) -> Workload:
    """The DiT-MoE variant with AdaLN-modulated blocks (Sec. 3), driven by a
    per-sample conditioning vector each step."""
    d = dit_variant(wl)
    return replace(d, name=d.name.replace("dit_", "ditada_", 1), adaln=True)


ADALN_WORKLOADS = {d.name: d for d in (adaln_variant(w) for w in WORKLOADS.values() if w.dtype == "bf16")}


def workload(name_or_index) -> Workload:
    if isinstance(name_or_index, int):
        return WORKLOADS[WORKLOAD_ORDER[name_or_index - 1]]
    if name_or_index in DIT_WORKLOADS:
        return DIT_WORKLOADS[name_or_index]
    if name_or_index in ADALN_WORKLOADS:
        return ADALN_WORKLOADS[name_or_index]
    return WORKLOADS[name_or_index]


# ---------------------------------------------------------------------------
# bf16 storage format
# ---------------------------------------------------------------------------

def round_to_bf16(a: np.ndarray) -> np.ndarray:
    """Round float32 values to the nearest bf16 (ties to even); returns float32.

    bf16 keeps the top 16 bits of an IEEE float32.  Inputs here are finite.
    """
    a = np.ascontiguousarray(a, dtype=np.float32)
    u = a.view(np.uint32).astype(np.uint64)
    lsb = (u >> 16) & 1
    u = (u + 0x7FFF + lsb) & 0xFFFF0000
    return u.astype(np.uint32).view(np.float32)


def bf16_bits(a: np.ndarray) -> np.ndarray:
    """The uint16 bit patterns of values that are already bf16-exact."""
    a = np.ascontiguousarray(a, dtype=np.float32)
    return (a.view(np.uint32) >> 16).astype(np.uint16)


def from_bf16_bits(b: np.ndarray) -> np.ndarray:
    return (np.ascontiguousarray(b, dtype=np.uint16).astype(np.uint32) << 16).view(np.float32)


def _store(wl: Workload, a: np.ndarray) -> np.ndarray:
    return round_to_bf16(a) if wl.dtype == "bf16" else np.ascontiguousarray(a, dtype=np.float32)


def _rng(*key) -> np.random.Generator:
    return np.random.Generator(np.random.PCG64(list(key)))


# ---------------------------------------------------------------------------
# Weights
# ---------------------------------------------------------------------------

def _skew_bias(wl: Workload) -> np.ndarray | None:
    """Router bias that makes top-k loads follow ``wl.router_skew`` at step 0.

    Only the 4:2:1:1 top-2 shape over 4 experts is needed: expert 0 is picked by
    every token (load T), expert 1 by half of them, experts 2 and 3 by a quarter
    each.  The logit of one expert for an N(0,1) token is N(b_e, s^2) with
    s = 0.02*sqrt(D).  Expert 0 gets b_0 = 6s; b_1 = d*s with d solving
    P(X1 > max(X2, X3)) = 1/2 for X1 ~ N(d,1), X2, X3 ~ N(0,1), i.e.
    integral phi(x - d) Phi(x)^2 dx = 1/2, solved by bisection on a quadrature.
    """
    if not wl.router_skew:
        return None
    if tuple(wl.router_skew) != (4, 2, 1, 1) or wl.top_k != 2 or wl.n_experts != 4:
        raise ValueError("only the 4:2:1:1 top-2 skew over 4 experts is defined")
    from scipy.special import ndtr
    x = np.linspace(-12.0, 12.0, 24001)
    dx = x[1] - x[0]

    def p_first(d):
        phi = np.exp(-0.5 * (x - d) ** 2) / math.sqrt(2.0 * math.pi)
        return float(np.sum(phi * ndtr(x) ** 2) * dx)

    lo, hi = 0.0, 4.0
    for _ in range(60):
        mid = 0.5 * (lo + hi)
        if p_first(mid) < 0.5:
            lo = mid
        else:
            hi = mid
    s = 0.02 * math.sqrt(wl.hidden)
    return np.array([6.0 * s, 0.5 * (lo + hi) * s, 0.0, 0.0], dtype=np.float32)


def make_layer_weights(wl: Workload, layer: int) -> dict:
    """Weights of one layer, all N(0, 0.02^2), stored in the workload dtype.

    Layout (row-major, "K-major" for both GEMMs of an expert):
      w_gate [E, D], b_gate [E] float32 or None,
      w1 [E, F, D] (first projection, rows are output features),
      w2 [E, D, F] (second projection),
      ws1 [S, F, D], ws2 [S, D, F] for S shared experts (absent when S = 0).
    """
    seed = _WEIGHT_SEED + wl.index
    E, D, F, S = wl.n_experts, wl.hidden, wl.ffn, wl.n_shared
    out = {}
    out["w_gate"] = _store(wl, 0.02 * _rng(seed, layer, _T_GATE).standard_normal((E, D), dtype=np.float32))
    out["b_gate"] = _skew_bias(wl)
    out["w1"] = _store(wl, 0.02 * _rng(seed, layer, _T_W1).standard_normal((E, F, D), dtype=np.float32))
    out["w2"] = _store(wl, 0.02 * _rng(seed, layer, _T_W2).standard_normal((E, D, F), dtype=np.float32))
    if S:
        out["ws1"] = _store(wl, 0.02 * _rng(seed, layer, _T_WS1).standard_normal((S, F, D), dtype=np.float32))
        out["ws2"] = _store(wl, 0.02 * _rng(seed, layer, _T_WS2).standard_normal((S, D, F), dtype=np.float32))
    else:
        out["ws1"] = out["ws2"] = None
    return out


def make_attn_weights(wl: Workload, layer: int) -> dict:
    """Attention weights of one DiT block, all N(0, 0.02^2), matrices in the
    workload dtype and biases float32:
      w_qkv [3D, D] (query, key, value projections stacked, heads contiguous
      within each), b_qkv [3D], w_o [D, D], b_o [D]."""
    seed = _WEIGHT_SEED + wl.index
    D = wl.hidden
    return {
        "w_qkv": _store(wl, 0.02 * _rng(seed, layer, _T_QKV).standard_normal((3 * D, D), dtype=np.float32)),
        "b_qkv": (0.02 * _rng(seed, layer, _T_BQKV).standard_normal(3 * D)).astype(np.float32),
        "w_o": _store(wl, 0.02 * _rng(seed, layer, _T_WO).standard_normal((D, D), dtype=np.float32)),
        "b_o": (0.02 * _rng(seed, layer, _T_BO).standard_normal(D)).astype(np.float32),
    }


def make_adaln_weights(wl: Workload, layer: int) -> dict:
    """AdaLN projection of one block, N(0, 0.02^2): w_ada [6D, D] in the
    workload dtype, b_ada [6D] float32."""
    seed = _WEIGHT_SEED + wl.index
    D = wl.hidden
    return {
        "w_ada": _store(wl, 0.02 * _rng(seed, layer, _T_ADA).standard_normal((6 * D, D), dtype=np.float32)),
        "b_ada": (0.02 * _rng(seed, layer, _T_BADA).standard_normal(6 * D)).astype(np.float32),
    }


def workload_conditioning(wl: Workload, n_steps: int | None = None) -> np.ndarray:
    """Per-step conditioning [n_steps, batch, D] of an AdaLN workload."""
    return conditioning(_TRAJ_SEED + wl.index, wl.batch, wl.hidden, wl.n_steps if n_steps is None else n_steps)


def tiny_attn(seed: int, D: int, dtype: str = "f32", bias: bool = True, wscale: float = 0.2) -> dict:
    """Small random attention weights for pins and parity cases."""
    rng = _rng(7500 + seed)
    st = round_to_bf16 if dtype == "bf16" else (lambda a: np.asarray(a, np.float32))
    return {
        "w_qkv": st(wscale * rng.standard_normal((3 * D, D), dtype=np.float32)),
        "b_qkv": (0.1 * rng.standard_normal(3 * D)).astype(np.float32) if bias else None,
        "w_o": st(wscale * rng.standard_normal((D, D), dtype=np.float32)),
        "b_o": (0.1 * rng.standard_normal(D)).astype(np.float32) if bias else None,
    }


def tiny_adaln(seed: int, D: int, dtype: str = "f32", wscale: float = 0.2, bias: bool = True) -> dict:
    """Small random AdaLN projection of one block: w_ada [6D, D] in the given
    dtype, b_ada [6D] float32 (or None)."""
    rng = _rng(7700 + seed)
    st = round_to_bf16 if dtype == "bf16" else (lambda a: np.asarray(a, np.float32))
    return {
        "w_ada": st(wscale * rng.standard_normal((6 * D, D), dtype=np.float32)),
        "b_ada": (0.1 * rng.standard_normal(6 * D)).astype(np.float32) if bias else None,
    }


def conditioning(seed: int, n_samples: int, D: int, n_steps: int) -> np.ndarray:
    """Per-step, per-sample conditioning vectors c [n_steps, n_samples, D]
    (float32) standing in for timestep + class embeddings: a fixed class part
    ~ N(0, 1) per sample plus a timestep part that varies smoothly with the
    step, sinusoids of the step index at D / 2 geometric frequencies."""
    rng = _rng(7900 + seed)
    cls = rng.standard_normal((n_samples, D)).astype(np.float64)
    half = D // 2
    freq = np.exp(-math.log(1000.0) * np.arange(half) / max(half, 1))
    out = np.empty((n_steps, n_samples, D), np.float32)
    for t in range(n_steps):
        ang = (n_steps - t) * 4.0 * freq
        emb = np.concatenate([np.cos(ang), np.sin(ang), np.zeros(D - 2 * half)])
        out[t] = (cls + emb[None, :]).astype(np.float32)
    return out


# ---------------------------------------------------------------------------
# Trajectories of the first layer's input
# ---------------------------------------------------------------------------

def trajectory(wl: Workload, n_steps: int | None = None, seed_offset: int = 0):
    """Yield the stack input x_t [T, D] (float32, bf16-exact for bf16) per step.

    x_0 ~ N(0, 1).  Drift models:
      "per_token": x_t = x_{t-1} + sigma_i * N(0, 1), sigma_i ~ U(0.01, 0.2).
      "decay":     x_t = x_{t-1} + sigma_t * a_i * b_d * N(0, 1), sigma_t linear
                   from 0.2 (t = 1) to 0.02 (last step), a_i and b_d ~ LogNormal(0, 0.5).
    The walk is kept in float32 and only the yielded copy is rounded.
    """
    n = wl.n_steps if n_steps is None else n_steps
    T, D = wl.n_tokens, wl.hidden
    rng = _rng(_TRAJ_SEED + wl.index, seed_offset)
    x = rng.standard_normal((T, D), dtype=np.float32)
    if wl.drift == "per_token":
        sig = rng.uniform(0.01, 0.2, size=(T, 1)).astype(np.float32)
        scale = lambda t: sig  # noqa: E731
    else:
        a = rng.lognormal(0.0, 0.5, size=(T, 1)).astype(np.float32)
        b = rng.lognormal(0.0, 0.5, size=(1, D)).astype(np.float32)
        ab = a * b
        last = max(n - 1, 1)

        def scale(t):
            s = 0.2 + (0.02 - 0.2) * (t - 1) / max(last - 1, 1)
            return np.float32(s) * ab
    for t in range(n):
        if t > 0:
            x = x + scale(t) * rng.standard_normal((T, D), dtype=np.float32)
        yield _store(wl, x)


def tiny_layer(seed: int, T: int, D: int, E: int, k: int, F: int, n_shared: int = 0,
               dtype: str = "f32", bias: bool = False, wscale: float = 0.2) -> tuple:
    """Small random layer for brute-force and parity cases: (weights, x0, rng)."""
    rng = _rng(7000 + seed)
    st = round_to_bf16 if dtype == "bf16" else (lambda a: np.asarray(a, np.float32))
    w = {
        "w_gate": st(wscale * rng.standard_normal((E, D), dtype=np.float32)),
        "b_gate": (0.1 * rng.standard_normal(E)).astype(np.float32) if bias else None,
        "w1": st(wscale * rng.standard_normal((E, F, D), dtype=np.float32)),
        "w2": st(wscale * rng.standard_normal((E, D, F), dtype=np.float32)),
        "ws1": st(wscale * rng.standard_normal((n_shared, F, D), dtype=np.float32)) if n_shared else None,
        "ws2": st(wscale * rng.standard_normal((n_shared, D, F), dtype=np.float32)) if n_shared else None,
    }
    x0 = st(rng.standard_normal((T, D), dtype=np.float32))
    return w, x0, rng


def make_layer_weights_device(wl: Workload, layer: int, device) -> dict:
    """The layer's weights drawn on the GPU with torch's seeded generator.

    Same distribution and layout as ``make_layer_weights`` (N(0, 0.02^2),
    rounded to the workload dtype) but drawn by torch's CUDA generator, which
    makes the multi-GB stacks in seconds.  The values differ from the numpy
    draw; a CPU consumer (the timed oracle baseline) copies them back.
    """
    import torch
    dt = torch.bfloat16 if wl.dtype == "bf16" else torch.float32
    E, D, F, S = wl.n_experts, wl.hidden, wl.ffn, wl.n_shared
    seed = (_WEIGHT_SEED + wl.index) * 1_000_003 + layer * 1009

    def draw(tid, shape):
        g = torch.Generator(device=device)
        g.manual_seed(seed + tid)
        t = torch.empty(shape, dtype=torch.float32, device=device)
        t.normal_(0.0, 0.02, generator=g)
        return t.to(dt).contiguous()

    out = {"w_gate": draw(_T_GATE, (E, D)), "w1": draw(_T_W1, (E, F, D)), "w2": draw(_T_W2, (E, D, F))}
    if wl.n_heads:
        out["w_qkv"] = draw(_T_QKV, (3 * D, D))
        out["b_qkv"] = draw(_T_BQKV, (3 * D,)).float()
        out["w_o"] = draw(_T_WO, (D, D))
        out["b_o"] = draw(_T_BO, (D,)).float()
    if wl.adaln:
        out["w_ada"] = draw(_T_ADA, (6 * D, D))
        out["b_ada"] = draw(_T_BADA, (6 * D,)).float()
    b = _skew_bias(wl)
    out["b_gate"] = None if b is None else torch.from_numpy(b).to(device)
    if S:
        out["ws1"] = draw(_T_WS1, (S, F, D))
        out["ws2"] = draw(_T_WS2, (S, D, F))
    else:
        out["ws1"] = out["ws2"] = None
    return out
